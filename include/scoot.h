/*
 * scoot.h - C ABI of the GB300 candidate-scoring path of SCOOT
 * (SLO-oriented tuning of LLM inference engines by Bayesian optimisation).
 *
 * One suggestion round scores a pool of N candidate engine configurations:
 *
 *   scoot_prune          known constraints, Eq. (2)
 *   scoot_rf_predict     random-forest probability of feasibility, Eq. (3)
 *   scoot_gp_posterior   GP posterior mean and variance (Section 4.3)
 *   scoot_gp_prepare_device  the GP state (fp64 factorisation) on the device
 *   scoot_gp_mle         GP hyperparameters by maximum likelihood (Section 4.3)
 *   scoot_acq_ei         expected improvement, Eq. (6)
 *   scoot_acq_ehvi       Monte-Carlo expected hypervolume improvement, Eq. (7)
 *   scoot_score_ei       posterior + EI in one pass
 *   scoot_score_ehvi     posterior + EHVI in one kernel
 *   scoot_score_ehvi_exact  posterior + exact EHVI (independent Gaussians)
 *   scoot_select_topq    top-q for parallel suggestion (Section 4.7)
 *   scoot_score_mace     posterior + UCB, PI, EI for MACE (Section 4.5)
 *   scoot_select_pareto  random k-subset of the (UCB, PI, EI) front (Section 4.7)
 *   scoot_sobol_configs  Sobol configurations (initial design, shortfall fill)
 *   scoot_rf_train       CART training of the feasibility forest (Algorithm 1)
 *
 * plus host-side preparation of per-round state (Cholesky factor of the
 * observations' covariance, box decomposition of the non-dominated region,
 * forest packing), all three in one call by scoot_round_state_build.
 *
 * Conventions
 *  - Every call returns a scoot_status: SCOOT_OK (0) or a negative error.
 *    No call aborts, throws across the ABI or traps on the device.  After an
 *    error, scoot_last_error(ctx) returns a message owned by the context.
 *  - Pointers named h_* are host memory; every other array pointer is device
 *    memory of the context's device.  All arrays are owned by the caller;
 *    the library owns only the workspace inside a scoot_ctx.
 *  - Device calls are asynchronous on the given stream (a cudaStream_t passed
 *    as void*; NULL is the legacy default stream).  Host-side calls
 *    (*_layout_init, *_prepare, *_build, *_pack) are synchronous and touch
 *    no device.
 *  - Candidates are stored structure-of-arrays: column p of a pool of n
 *    candidates with leading dimension ld is cand[p * ld + i], one 32-bit
 *    word per parameter: integer and categorical parameters as int32,
 *    continuous ones as float32 bit patterns.  cand must be 16-byte aligned
 *    and ld a multiple of 4 with ld >= n.
 *  - Objectives are maximised (Eq. 1 with the lambda signs applied).
 *  - A context is used by one host thread at a time.  Calls on one context
 *    that overlap on the GPU share its workspace: order them on one stream.
 */
#ifndef SCOOT_H
#define SCOOT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t scoot_status;
#define SCOOT_OK            0
#define SCOOT_EINVAL       -1   /* bad argument: null, size, alignment, NaN, malformed input */
#define SCOOT_ENOMEM       -2   /* workspace allocation failed */
#define SCOOT_ECUDA        -3   /* a CUDA runtime call failed */
#define SCOOT_EDEVICE      -4   /* a kernel flagged a bad index or value at run time */
#define SCOOT_ETIMEOUT     -5   /* a bounded device-side wait gave up */
#define SCOOT_EUNSUPPORTED -6   /* size or option beyond what the library handles */

/* Parameter kinds of the mixed search space (Section 3, Table 1). */
#define SCOOT_INT_UNIFORM 0
#define SCOOT_INT_LOG     1
#define SCOOT_CATEGORICAL 2   /* booleans are categoricals of two */
#define SCOOT_CONTINUOUS  3

/* Covariance functions (Section 4.3 names Matern-3/2; Matern-5/2 ARD is the default). */
#define SCOOT_MATERN52 0
#define SCOOT_MATERN32 1

#define SCOOT_MAX_DIM      16   /* parameters per configuration */
#define SCOOT_MAX_CLAUSES  16   /* known-constraint clauses per call */
#define SCOOT_MAX_OBJ       4   /* objectives */
#define SCOOT_MAX_OBS     640   /* observed configurations: the posterior kernels hold a
                                      64-candidate tile's covariance rows (n x 64 fp32) and the
                                      observations in shared memory (227 KB) */
#define SCOOT_MAX_Q        64   /* picks per top-q call */

/* One parameter: kind, number of categories (categorical only) and the
 * range [lo, hi] (integer and continuous kinds).  16 bytes. */
typedef struct {
    int32_t kind;
    int32_t n_choices;
    float lo;
    float hi;
} scoot_param;

/* One known constraint (Eq. 2): if x[guard_param[g]] == guard_value[g] for
 * every g < n_guard, then sum_{t < n_term} coef[t] * x[term_param[t]] >= rhs
 * must hold, evaluated exactly in 64-bit integers.  Only integer and
 * categorical parameters may appear.  80 bytes. */
typedef struct {
    int32_t n_guard;
    int32_t guard_param[2];
    int32_t guard_value[2];
    int32_t n_term;
    int32_t term_param[4];
    int64_t coef[4];
    int64_t rhs;
} scoot_clause;

/* One regression-tree node, 8 bytes.  A split node (flags & 1 == 0) sends a
 * configuration to node `left` when x[feat] <= val and to node left + 1
 * otherwise; child indices count from the tree's first node.  A leaf
 * (flags & 1) carries an integer vote count in val, 0 <= val <= leaf_scale.
 * x[feat] is the stored value as a float (integers and category indices
 * converted exactly, continuous values as stored). */
typedef struct {
    float val;
    uint16_t left;
    uint8_t feat;
    uint8_t flags;
} scoot_node;

typedef struct scoot_ctx scoot_ctx;

/* ------------------------------------------------------------------ context */

/* Create a context on CUDA device `device` (made current for every call on
 * the context).  *out receives the handle; on error *out is NULL. */
scoot_status scoot_ctx_create(int32_t device, scoot_ctx** out);
scoot_status scoot_ctx_destroy(scoot_ctx* ctx);
/* Message of the last error on ctx ("" if none).  Owned by ctx. */
const char* scoot_last_error(const scoot_ctx* ctx);
const char* scoot_status_string(scoot_status s);
/* Wait for `stream`, then read and clear the context's device error word:
 * SCOOT_EDEVICE if a kernel flagged a bad index or value since the last
 * check, SCOOT_ETIMEOUT if a bounded wait gave up, SCOOT_EUNSUPPORTED if a
 * Pareto filter ran out of survivor capacity, SCOOT_EINVAL if a kernel met a
 * non-finite input it had to validate, else SCOOT_OK. */
scoot_status scoot_ctx_check(scoot_ctx* ctx, void* stream);
/* Bytes of device workspace the context currently holds. */
scoot_status scoot_ctx_workspace_bytes(const scoot_ctx* ctx, int64_t* bytes);

/* Phase timing, a measurement aid (off by default).  With enable != 0 the
 * calls that launch several kinds of kernel (scoot_suggest_fantasy) record a
 * CUDA event on their stream before their first launch and after each
 * launch, up to SCOOT_MAX_MARKS launches per call; scoot_ctx_phase_times
 * waits for the last timed call's events and returns, per launch in order,
 * its kind (SCOOT_PHASE_*) in h_kind and its milliseconds in h_ms (at most
 * cap entries; *count = the number of timed launches).  Leave it off for
 * calls captured in a CUDA graph. */
#define SCOOT_MAX_MARKS          256
#define SCOOT_PHASE_COMPACT        0   /* compaction of the live candidates */
#define SCOOT_PHASE_POSTERIOR      1   /* posterior with the whitened rows V */
#define SCOOT_PHASE_FANT_INIT      2   /* the observations' front and boxes */
#define SCOOT_PHASE_FANT_PASS      3   /* a pick's pass: downdate, EHVI, block argmax */
#define SCOOT_PHASE_FANT_PICK      4   /* a pick's fp64 terms, front and boxes */
#define SCOOT_PHASE_SCATTER        5   /* variances scattered to var_out */
scoot_status scoot_ctx_set_timing(scoot_ctx* ctx, int32_t enable);

/* Tensor cores for the posterior (on by default).  With enable != 0 the
 * posterior of scoot_gp_posterior, scoot_score_ei, scoot_score_mace and
 * scoot_suggest_fantasy / scoot_fantasy_begin computes
 * V = L^{-1} k(X, x) on the tcgen05 tensor cores when the padded observation
 * count is at most 256 and the state fits a block's shared memory: each fp32
 * operand split into three bf16 parts, six part products accumulated in fp32
 * (the m l, l m, l l products, of order 2^-24, dropped); with enable == 0,
 * or outside those limits, the fp32 SIMT product.  The paper has no
 * counterpart (Section 4.3 states the posterior, not how it is computed). */
scoot_status scoot_ctx_set_tensor_cores(scoot_ctx* ctx, int32_t enable);
scoot_status scoot_ctx_phase_times(scoot_ctx* ctx, int32_t cap, int32_t* h_kind, float* h_ms, int32_t* count);

/* ------------------------------------------------------------------ 1. prune, Eq. (2) */

/* mask[i] = 1 when candidate i satisfies every clause of h_clauses, else 0
 * (the solution space pruned by known constraints, Section 4.5).  Only the
 * columns named by some clause are read.  If n_feasible is not NULL it is a
 * device int64 that receives the number of feasible candidates (overwritten,
 * not accumulated).  n == 0 is valid and writes nothing but the count. */
scoot_status scoot_prune(scoot_ctx* ctx, const scoot_param* h_space, int32_t d,
                         const scoot_clause* h_clauses, int32_t n_clauses,
                         const uint32_t* cand, int64_t n, int64_t ld,
                         uint8_t* mask, int64_t* n_feasible, void* stream);

/* ------------------------------------------------------------------ 2. random forest, Eq. (3) */

/* Packed forest: a device blob built by scoot_forest_pack. */
typedef struct {
    int32_t n_trees;
    int32_t n_nodes;          /* total nodes */
    int32_t d;                /* features */
    int32_t leaf_scale;       /* V: leaves hold votes in [0, V] */
    int32_t max_depth;        /* longest root-to-leaf path (edges) */
    int32_t n_chunks;         /* groups of whole trees staged in shared memory one at a time */
    int32_t max_chunk_nodes;  /* nodes of the largest group */
    int32_t reserved;
    int64_t bytes;            /* blob size */
    int64_t off_chunks;       /* int32[n_chunks][4]: first tree, tree count, first node, node count */
    int64_t off_roots;        /* int32[n_trees]: first node of each tree */
    int64_t off_nodes;        /* scoot_node[n_nodes], split nodes' left child counted from the
                                 first node of their chunk */
} scoot_forest_layout;

/* Validate a forest given as nodes plus tree offsets (tree t owns nodes
 * h_tree_offset[t] .. h_tree_offset[t+1]-1) and plan its blob.  Rejects
 * child indices outside the tree or not after their parent (so no cycles),
 * features >= d, and leaf votes that are not integers in [0, leaf_scale]. */
scoot_status scoot_forest_layout_init(const scoot_node* h_nodes, const int32_t* h_tree_offset,
                                      int32_t n_trees, int32_t d, int32_t leaf_scale,
                                      scoot_forest_layout* out);
/* Write the blob (layout->bytes bytes) into h_blob; copy it to the device as is. */
scoot_status scoot_forest_pack(const scoot_forest_layout* layout, const scoot_node* h_nodes,
                               const int32_t* h_tree_offset, void* h_blob);

/* votes[i] = sum over trees of the leaf votes reached by candidate i, for
 * every candidate with mask[i] == 1 on entry; then mask[i] &= (delta_den *
 * votes[i] >= delta_num * leaf_scale * n_trees), i.e. POF(x) >= Delta with
 * POF = votes / (leaf_scale * T) and Delta = delta_num / delta_den (Eq. 3).
 * Candidates with mask[i] == 0 on entry are not walked: votes[i] = 0.
 * mask may be NULL (every candidate walked, no mask written).  n_feasible,
 * if not NULL, is a device int64 receiving the count of mask == 1 after. */
scoot_status scoot_rf_predict(scoot_ctx* ctx, const scoot_forest_layout* layout,
                              const void* forest, const scoot_param* h_space,
                              const uint32_t* cand, int64_t n, int64_t ld,
                              uint32_t delta_num, uint32_t delta_den,
                              uint32_t* votes, uint8_t* mask, int64_t* n_feasible,
                              void* stream);

/* ------------------------------------------------------------------ 3. GP posterior (Section 4.3) */

/* Per-round GP state for M objectives over n observations: a device blob
 * built on the host by scoot_gp_prepare (fp64 Cholesky of K + tau^2 I, then
 * alpha = (K + tau^2 I)^{-1} Y and L^{-1}, stored in fp32). */
typedef struct {
    int32_t n, d, n_obj, kernel;
    int32_t n_rb;             /* row blocks of 64 in the tiled L^{-1} */
    int32_t n_tiles;          /* 32 x 64 tiles of L^{-1} per objective */
    int32_t n_ord;            /* ordinal (integer or continuous) parameters */
    int32_t n_pat;            /* joint category patterns: product of the categoricals' n_choices (1 if none) */
    int64_t bytes;
    int64_t off_fmap;         /* float[d][4]: kind, a, b, source parameter of each feature, ordinal
                                 parameters first, then categorical ones ("feature order"); for a
                                 categorical feature a = n_choices and b = its mixed-radix stride */
    int64_t off_xs;           /* float[M][n][d]: observed features in feature order, ordinal ones
                                 scaled by 1/lengthscale, categorical ones as the category index */
    int64_t off_ils;          /* float[M][d]: 1/l (ordinal) or 1/l^2 (categorical), feature order */
    int64_t off_alpha;        /* float[M][n] */
    int64_t off_linv;         /* float[M][n_tiles][32][64]: L^{-1} tiles, transposed, zero-filled */
    int64_t off_scal;         /* float[M][4]: signal variance, noise variance, best observed y,
                                 1 if the objective's ordinal features are warped else 0 */
    int64_t off_cat;          /* float[M][n][n_pat]: for each category pattern p (mixed radix over the
                                 categorical parameters in feature order), sum_c [p_c != X_jc] / l_c^2 */
    int64_t off_warp;         /* float[M][d][2]: Kumaraswamy (a, b) per feature, feature order
                                 (1, 1 when not warped) */
} scoot_gp_layout;

/* Plan the blob for n observations of the d-parameter space h_space, M
 * objectives and a covariance kernel.  SCOOT_EUNSUPPORTED if the categorical
 * parameters have more than 4096 joint patterns. */
scoot_status scoot_gp_layout_init(const scoot_param* h_space, int32_t n, int32_t d, int32_t n_obj, int32_t kernel,
                                  scoot_gp_layout* out);
/* Build the blob on the host.  h_x_obs: observed configurations, SoA words
 * [d][ld_obs]; h_y: standardised observed values [M][n]; h_lengthscale
 * [M][d] (> 0); h_signal_var, h_noise_var [M] (> 0 and >= 0).  Features
 * (the covariance's input coordinates): integer log-uniform parameters
 * (ln v - ln lo)/(ln hi - ln lo); integer uniform and continuous ones
 * (v - lo)/(hi - lo); categoricals compared for equality, adding
 * [c != c']/l^2 to r^2.  Fails with SCOOT_EINVAL if K + tau^2 I is not
 * numerically positive definite.  If h_cond is not NULL it receives, per
 * objective, the ratio of the largest to the smallest pivot squared of the
 * Cholesky factor (a cheap conditioning indicator). */
scoot_status scoot_gp_prepare(const scoot_param* h_space, const uint32_t* h_x_obs, int64_t ld_obs,
                              const float* h_y, const float* h_lengthscale,
                              const float* h_signal_var, const float* h_noise_var,
                              const scoot_gp_layout* layout, void* h_blob, double* h_cond);

/* scoot_gp_prepare with input warping (the kernel of Section 4.3 is Matérn
 * with input warping): every ordinal feature u of objective m is replaced by
 * the Kumaraswamy CDF w(u) = 1 - (1 - u^a)^b before distances are taken, for
 * the observations here and for the candidates inside the posterior and
 * scoring kernels.  h_warp: [M][d][2] = (a, b) per parameter (source order,
 * a, b > 0 and finite; entries of categorical parameters are ignored).  The
 * kernels evaluate w as -expm1(b log1p(-u^a)).  scoot_suggest_fantasy does
 * not take warped states (SCOOT_EUNSUPPORTED). */
scoot_status scoot_gp_prepare_warped(const scoot_param* h_space, const uint32_t* h_x_obs, int64_t ld_obs,
                                     const float* h_y, const float* h_lengthscale,
                                     const float* h_signal_var, const float* h_noise_var,
                                     const float* h_warp, const scoot_gp_layout* layout, void* h_blob,
                                     double* h_cond);

/* Bytes of device scratch scoot_gp_prepare_device needs for a layout:
 * 8 M (n d + n (n + 1) / 2), and another 8 M n (n + 1) / 2 when n > 160. */
scoot_status scoot_gp_device_work_bytes(const scoot_gp_layout* layout, int64_t* bytes);

/* scoot_gp_prepare (h_warp NULL) or scoot_gp_prepare_warped on the device,
 * into a device blob of the same layout, asynchronously on `stream`: the
 * features, K + tau^2 I and its Cholesky factorisation in fp64, L^{-1} formed
 * by applying the factorisation's elimination to the identity, alpha, and
 * the same fp32 tables.  Device inputs: obs (words [d][ld_obs]), y [M][n],
 * lengthscale [M][d], signal_var [M], noise_var [M], warp [M][d][2] or NULL
 * (the conventions of scoot_gp_prepare_warped); blob (layout->bytes,
 * 16-byte aligned); work: caller-owned scratch of at least
 * scoot_gp_device_work_bytes bytes, 16-byte aligned, not used by other work
 * in flight (the context's workspace is not touched, so CUDA graphs captured
 * on the context stay valid).  A non-finite or out-of-range input, or a
 * matrix that is not numerically positive definite, makes scoot_ctx_check
 * return SCOOT_EINVAL and leaves the blob undefined.  The conditioning
 * indicator of the host function is not computed. */
scoot_status scoot_gp_prepare_device(scoot_ctx* ctx, const scoot_param* h_space, const scoot_gp_layout* layout,
                                     const uint32_t* obs, int64_t ld_obs, const float* y, const float* lengthscale,
                                     const float* signal_var, const float* noise_var, const float* warp,
                                     void* blob, void* work, int64_t work_bytes, void* stream);

/* GP hyperparameters by maximum likelihood (Section 4.3 learns tau^2 this
 * way), for every objective m and start s at once on the device.  theta =
 * (ln l_1 .. ln l_d, ln s_f^2, ln tau^2), P = d + 2 values; the log marginal
 * likelihood of the zero-mean GP with covariance s_f^2 k(r) + tau^2 I over
 * the n observations (features as in scoot_gp_prepare, no warping) is
 *   lml = -y^T K^{-1} y / 2 - log det K / 2 - n log(2 pi) / 2
 * with gradient d lml / d theta_p = tr((alpha alpha^T - K^{-1}) dK/dtheta_p) / 2.
 * From theta0 [S][M][P] (device, fp64) each (s, m) takes `steps` projected
 * Adam ascent steps (beta1 0.9, beta2 0.999, eps 1e-8; step size
 * lr (1 - t / steps) at step t; theta clipped to [h_lo, h_hi] (host [P])
 * after each step; parameter p moves only if bit p of free_mask is set).
 * Outputs (device, fp64): theta [S][M][P] after the last step, lml [S][M]
 * there (-inf if K + tau^2 I stopped being positive definite, theta then
 * being the last good one) and, if grad is not NULL, the gradient there
 * [S][M][P].  obs: words [d][ld_obs]; y: [M][n] float32.  work: scratch of
 * scoot_gp_mle_work_bytes bytes, 16-byte aligned.  S * M <= 65535.  A
 * non-finite feature or y makes scoot_ctx_check return SCOOT_EINVAL. */
scoot_status scoot_gp_mle(scoot_ctx* ctx, const scoot_param* h_space, int32_t d, const uint32_t* obs, int64_t ld_obs,
                          int32_t n, const float* y, int32_t n_obj, int32_t kernel, const double* theta0,
                          int32_t n_starts, const double* h_lo, const double* h_hi, uint32_t free_mask, int32_t steps,
                          double lr, double* theta, double* lml, double* grad, void* work, int64_t work_bytes,
                          void* stream);
scoot_status scoot_gp_mle_work_bytes(int32_t n, int32_t d, int32_t n_obj, int32_t n_starts, int64_t* bytes);

/* One device buffer for scoot_gp_prepare_device_from_host: the uploaded
 * inputs (upload_bytes), the blob at blob_off, the scratch at work_off;
 * total_bytes in all (256-byte aligned parts). */
scoot_status scoot_gp_device_buffer_layout(const scoot_gp_layout* layout, int32_t warped, int64_t* upload_bytes,
                                           int64_t* blob_off, int64_t* work_off, int64_t* total_bytes);
/* scoot_gp_prepare_device from host inputs (the arguments of
 * scoot_gp_prepare_warped; h_warp may be NULL): packs them into h_stage
 * (pinned host memory of at least upload_bytes, free to reuse once `stream`
 * has passed this call), copies them to the start of buf (device,
 * total_bytes of scoot_gp_device_buffer_layout) and launches the device
 * build into buf + blob_off, all asynchronously on `stream`. */
scoot_status scoot_gp_prepare_device_from_host(scoot_ctx* ctx, const scoot_param* h_space, const scoot_gp_layout* layout,
                                               const uint32_t* h_x_obs, int64_t ld_obs, const float* h_y,
                                               const float* h_lengthscale, const float* h_signal_var,
                                               const float* h_noise_var, const float* h_warp, void* h_stage,
                                               void* buf, int64_t buf_bytes, void* stream);

/* mean[m * ldo + i], var[m * ldo + i] for every candidate i < n and
 * objective m:  mu = k(x, X)(K + tau^2 I)^{-1} Y and
 * sigma^2 = k(x, x) - k(x, X)(K + tau^2 I)^{-1} k(X, x) (latent f, clamped
 * at 0).  If mask is not NULL, candidates with mask[i] == 0 are skipped and
 * their outputs left untouched.  ldo >= n. */
scoot_status scoot_gp_posterior(scoot_ctx* ctx, const scoot_gp_layout* layout, const void* state,
                                const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                                float* mean, float* var, int64_t ldo, void* stream);

/* ------------------------------------------------------------------ 4. acquisition */

/* EI(x) = E[max(0, f(x) + xi - y_best)] in closed form, Eq. (6):
 * a = mu - y_best + xi, z = a / sigma, EI = a Phi(z) + sigma phi(z);
 * EI = max(0, a) when sigma == 0.  acq[i] = -inf where mask[i] == 0
 * (mask may be NULL). */
scoot_status scoot_acq_ei(scoot_ctx* ctx, const float* mean, const float* var,
                          const uint8_t* mask, int64_t n, float y_best, float xi,
                          float* acq, void* stream);

/* Box decomposition of the region above h_ref that the Pareto front of the
 * points h_y ([M][n_pts], maximised) does not dominate.  Only points that
 * strictly dominate h_ref take part (others enclose no volume, Eq. 8).
 * Boxes are written row-major: h_lo[b * M + j], h_hi[b * M + j] (+inf where
 * unbounded); *n_boxes receives the count, *front_size the front's size.
 * cap is the capacity of h_lo / h_hi in boxes (SCOOT_EUNSUPPORTED if too
 * small; *n_boxes then holds the count needed).  2 <= M <= SCOOT_MAX_OBJ. */
scoot_status scoot_boxes_build(const float* h_y, int32_t n_pts, int32_t n_obj, const float* h_ref,
                               int32_t cap, float* h_lo, float* h_hi, int32_t* n_boxes,
                               int32_t* front_size);

/* Corner indices of boxes for the exact EHVI (scoot_acq_ehvi_exact,
 * scoot_score_ehvi_exact).  h_lo, h_hi: n_boxes boxes [B][M] as written by
 * scoot_boxes_build.  For each objective j, h_grid[j * grid_cap + g]
 * (g < h_n_grid[j]) receives the distinct finite box coordinates on that axis
 * in increasing order, and h_corner[b * M + j] = lo | hi << 16, the indices of
 * box b's lower and upper coordinates in that list (h_n_grid[j] standing for
 * +inf).  Host only.  SCOOT_EINVAL for a NaN, an infinite lower corner or
 * hi <= lo; SCOOT_EUNSUPPORTED if an axis has more than grid_cap (or 65535)
 * coordinates (h_n_grid then holds the counts found so far). */
scoot_status scoot_boxes_index(const float* h_lo, const float* h_hi, int32_t n_boxes, int32_t n_obj,
                               int32_t grid_cap, float* h_grid, int32_t* h_n_grid, uint32_t* h_corner);

/* Monte-Carlo EHVI, Eq. (7): with base samples eps [S][M] shared by every
 * candidate, y_s = mu + sigma * eps_s and
 * EHVI = (1/S) sum_s sum_b prod_j max(0, min(y_sj, hi_bj) - lo_bj)
 * over the n_boxes boxes (lo, hi: device, [B][M]).  mean/var as written by
 * scoot_gp_posterior ([M][ldm]).  acq[i] = -inf where mask[i] == 0. */
scoot_status scoot_acq_ehvi(scoot_ctx* ctx, const float* mean, const float* var, int64_t ldm,
                            int32_t n_obj, const uint8_t* mask, int64_t n,
                            const float* box_lo, const float* box_hi, int32_t n_boxes,
                            const float* eps, int32_t n_mc, float* acq, void* stream);

/* scoot_gp_posterior followed by scoot_acq_ei, in one pass, without
 * writing mean or variance (objective 0; y_best is the state's best
 * observed value of objective 0).  With the context's tensor cores on and
 * at most 256 observations the pass is the tensor-core posterior with an EI
 * epilogue (after a small kernel that splits L^{-1} into bf16 parts in the
 * context workspace), else one fused fp32 kernel; where mask[i] == 0,
 * acq[i] = -inf. */
scoot_status scoot_score_ei(scoot_ctx* ctx, const scoot_gp_layout* layout, const void* state,
                            const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                            float xi, float* acq, void* stream);

/* scoot_gp_posterior followed by scoot_acq_ehvi, in one kernel. */
scoot_status scoot_score_ehvi(scoot_ctx* ctx, const scoot_gp_layout* layout, const void* state,
                              const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                              const float* box_lo, const float* box_hi, int32_t n_boxes,
                              const float* eps, int32_t n_mc, float* acq, void* stream);

/* EHVI (Eq. 7) as the exact expectation over independent Gaussian
 * objectives Y_j ~ N(mu_j, sigma_j^2), the closed form behind the paper's
 * EHVI reference (Yang et al.):
 *   EHVI = sum_b prod_j [psi_j(lo_bj) - psi_j(hi_bj)],
 *   psi_j(a) = E[max(0, Y_j - a)] = sigma_j phi(z) + (mu_j - a) Phi(z),
 *   z = (mu_j - a) / sigma_j  (max(0, mu_j - a) when sigma_j = 0; 0 at +inf),
 * over boxes given as scoot_boxes_index writes them: grid (device
 * [M][grid_cap]), h_n_grid (host [M]), corner (device [B][M]).  psi is
 * evaluated once per grid coordinate and candidate.  mean/var as written by
 * scoot_gp_posterior ([M][ldm]); acq[i] = -inf where mask[i] == 0.
 * SCOOT_EUNSUPPORTED when sum_j (h_n_grid[j] + 1) > 320.  A corner index
 * beyond h_n_grid is clamped and flagged (SCOOT_EDEVICE from
 * scoot_ctx_check). */
scoot_status scoot_acq_ehvi_exact(scoot_ctx* ctx, const float* mean, const float* var, int64_t ldm,
                                  int32_t n_obj, const uint8_t* mask, int64_t n, const float* grid,
                                  int32_t grid_cap, const int32_t* h_n_grid, const uint32_t* corner,
                                  int32_t n_boxes, float* acq, void* stream);

/* scoot_gp_posterior followed by scoot_acq_ehvi_exact, in one kernel. */
scoot_status scoot_score_ehvi_exact(scoot_ctx* ctx, const scoot_gp_layout* layout, const void* state,
                                    const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                                    const float* grid, int32_t grid_cap, const int32_t* h_n_grid,
                                    const uint32_t* corner, int32_t n_boxes, float* acq, void* stream);

/* ------------------------------------------------------------------ a round's host state in one call */

/* Inputs of scoot_round_state_build (host arrays, conventions of the calls
 * it combines). */
typedef struct {
    const scoot_param* space;
    int32_t d;
    const uint32_t* x_obs;       /* observations, words [d][ld_obs] */
    int64_t ld_obs;
    int32_t n;                   /* observations */
    int32_t n_obj;               /* M */
    const float* y;              /* [M][n] */
    const float* lengthscale;    /* [M][d] */
    const float* signal_var;     /* [M] */
    const float* noise_var;      /* [M] */
    const float* warp;           /* [M][d][2] or NULL */
    int32_t kernel;
    int32_t gp_on_device;        /* 1: no GP state here (scoot_gp_prepare_device builds it) */
    const scoot_node* nodes;
    const int32_t* tree_offset;  /* [n_trees + 1] */
    int32_t n_trees;
    int32_t leaf_scale;
    int32_t boxes;               /* 0: none (EI, MACE); 1: boxes and eps (MC EHVI); 2: boxes and their grid index (exact EHVI) */
    const float* ref;            /* [M] (boxes != 0) */
    const float* eps;            /* [S][M] (boxes == 1) */
    int32_t n_mc;                /* S */
    int32_t grid_cap;            /* boxes == 2: coordinates per axis (0: 256) */
    int32_t fantasy_q;           /* > 0: also the fantasy state for this many picks (needs ref; no warp,
                                    gp_on_device 0) */
} scoot_round_inputs;

/* Where scoot_round_state_build put each part in the buffer (256-byte
 * aligned offsets; -1 for an absent part). */
typedef struct {
    int64_t bytes;               /* bytes used: the upload */
    int64_t off_gp, off_forest, off_box_lo, off_box_hi, off_eps, off_grid, off_corner;
    int64_t off_fant;            /* fantasy state (fantasy_q > 0) */
    int32_t fant_box_cap;        /* its box_cap */
    int32_t n_boxes, front_size;
    int32_t grid_cap;
    int32_t n_grid[SCOOT_MAX_OBJ];
    double cond[SCOOT_MAX_OBJ];  /* the GP factorisations' conditioning indicator */
    scoot_gp_layout gp;
    scoot_forest_layout forest;
} scoot_round_state;

/* A round's host-side state in one buffer h_buf (cap bytes, host): the GP
 * blob (scoot_gp_prepare_warped), the packed forest (scoot_forest_pack) and,
 * as asked, the boxes (scoot_boxes_build) with eps or with their grid index
 * (scoot_boxes_index), and the fantasy state (scoot_fantasy_prepare, from
 * the GP blob's own factorisation).  Copy the first out->bytes bytes to the
 * device as
 * they are.  The GP factorisation runs on a library worker thread while the
 * calling thread packs the forest and builds the boxes.  SCOOT_ENOMEM if
 * cap is too small (out->bytes then holds the size needed); the errors of
 * the calls it combines otherwise. */
scoot_status scoot_round_state_build(const scoot_round_inputs* in, void* h_buf, int64_t cap, scoot_round_state* out);

/* ------------------------------------------------------------------ 5. top-q (Section 4.7) */

/* The min(q, eligible) candidates with the largest acq, eligible meaning
 * mask[i] == 1 (mask may be NULL) and acq[i] neither NaN nor -inf.  Order:
 * value descending, then index ascending (the lowest index wins a tie).
 * idx (int64 [q]), val (float [q]) and count (int32 [1]) are device
 * outputs; entries beyond count are set to -1 / -inf.  1 <= q <= SCOOT_MAX_Q. */
scoot_status scoot_select_topq(scoot_ctx* ctx, const float* acq, const uint8_t* mask, int64_t n,
                               int32_t q, int64_t* idx, float* val, int32_t* count, void* stream);

/* ------------------------------------------------------------------ the tuning loop's sampling (Algorithm 1, Section 4.6) */

/* Points skip .. skip + n - 1 of a d-dimensional Sobol sequence mapped onto
 * the search space h_space and written as pool words cand [d][ld] (device):
 * the initial design of Algorithm 1 and the shortfall fill of Section 4.6
 * (both sample with a Sobol sequence).  Dimension 0 is the van der Corput
 * sequence; dimension j >= 1 uses the j-th primitive polynomial over GF(2)
 * (by degree, then by its middle coefficients as a binary number, the
 * highest-degree one most significant) with unit initial direction
 * integers.  With u = point / 2^32 in [0, 1), in fp64 with one rounding per
 * operation: integer log-uniform round(exp(ln lo + u (ln hi - ln lo)))
 * (half to even) clamped to [lo, hi]; integer uniform
 * min(lo + floor(u (hi - lo + 1)), hi); categorical floor(u n_choices);
 * continuous lo + u (hi - lo) rounded to float32.  skip + n <= 2^32 - 1. */
scoot_status scoot_sobol_configs(scoot_ctx* ctx, const scoot_param* h_space, int32_t d, int64_t skip, int64_t n,
                                 uint32_t* cand, int64_t ld, void* stream);

/* The first `need` positions p < n with mask[p] != 0, in increasing order
 * (the shortfall fill takes the first Sobol points that pass the known
 * constraints): idx (int64 [need], -1 beyond the count), count (int32 [1]).
 * 1 <= need <= SCOOT_MAX_Q, n < 2^31. */
scoot_status scoot_first_feasible(scoot_ctx* ctx, const uint8_t* mask, int64_t n, int32_t need, int64_t* idx,
                                  int32_t* count, void* stream);

/* beta_t, the UCB coefficient of tuning iteration t >= 1 (Section 4.5):
 * beta_t = 2 log(t^2 pi^2 / (6 delta)) with delta = 1 / t^2, taken as the
 * factor of sigma in UCB = mu + beta sigma, as printed (the kappa argument
 * of scoot_acq_mace / scoot_score_mace).  Host, synchronous. */
scoot_status scoot_ucb_beta(int32_t t, double* beta);

/* The observed objectives as the GP models them: per objective m,
 * h_y_std[m][i] = (h_y[m][i] - mean_m) / sd_m over the n observations
 * (population standard deviation, floored at 1e-12), computed in fp64
 * (Section 4.3 fits zero-mean GPs; the loop standardises before each fit).
 * If h_ref is not NULL, h_ref[m] = min_i h_y_std[m][i] - ref_margin: a
 * reference point below every observation (the loop's reading of the
 * default configuration's objectives, Section 4.5).  h_y, h_y_std [n_obj][n]
 * host; SCOOT_EINVAL on a non-finite value.  Host, synchronous. */
scoot_status scoot_standardize(const float* h_y, int32_t n_obj, int32_t n, float* h_y_std, float* h_ref,
                               float ref_margin);

/* Algorithm 1's feasibility-threshold controller after k suggestions were
 * evaluated (host): if any result was invalid, Delta becomes
 * min(0.75, max(0.5, Delta + 0.05)) and the count of feasible suggestions
 * is cleared; otherwise the count grows by k and, once it reaches 5, Delta
 * becomes max(0.25, Delta - 0.05) and the count loses 5. */
scoot_status scoot_delta_update(double* h_delta, int32_t* h_count, int32_t k, int32_t any_invalid);

#define SCOOT_RF_TRAIN_MAX_OBS 1024  /* observations and bootstrap size per tree */

/* Train the feasibility forest of Algorithm 1 (random forest regression of
 * the crash labels, Section 4.6): tree t is a CART regression tree on the
 * bootstrap sample boot[t * m + k], k < m (indices into the n observations;
 * int32, device).  obs holds the observations as pool words [d][ld]
 * (device; the features are their stored values as floats, as scoot_node's
 * x[feat]); labels (uint8 [n], device) are 1 for a feasible observation, 0
 * for a crash.
 * Growth is breadth first.  A node of m' samples with p positives becomes a
 * leaf at depth max_depth (the root has depth 0), when p is 0 or m', or when
 * all its samples share every feature value; a leaf stores
 * floor((2 leaf_scale p + m') / (2 m')) votes (leaf_scale p / m' rounded half
 * up).  Otherwise the node splits on "x[f] <= v", v one of its samples'
 * values of feature f other than the largest, minimising the squared error
 * of the two children p_l (m_l - p_l) / m_l + p_r (m_r - p_r) / m_r, compared
 * exactly; ties go to the lower f, then the lower v (-0 and +0 are one
 * value; a zero threshold is stored as +0).  The two children of a node are
 * numbered next to each other in breadth-first order.  work: caller-owned
 * device scratch of scoot_rf_train_work_bytes(n, d) bytes (the feature ranks
 * of the observations), 16-byte aligned.
 * Output: nodes (scoot_node [n_trees][node_cap], device), tree t in
 * nodes[t * node_cap ...] with child indices counted from its first node,
 * n_nodes (int32 [n_trees], device) its node count (<= 2 m - 1, so node_cap
 * >= 2 m - 1 is required).  Pass the compacted nodes to
 * scoot_forest_layout_init.  1 <= n, m <= SCOOT_RF_TRAIN_MAX_OBS, 1 <= d <=
 * SCOOT_MAX_DIM, 0 <= max_depth <= 255, 1 <= leaf_scale <= 2^24.  A
 * bootstrap index outside 0..n-1 (SCOOT_EDEVICE from scoot_ctx_check), or a
 * drawn observation with a non-finite feature or a label other than 0/1
 * (SCOOT_EINVAL from scoot_ctx_check), leaves that tree empty
 * (n_nodes[t] = 0). */
scoot_status scoot_rf_train(scoot_ctx* ctx, const scoot_param* h_space, int32_t d, const uint32_t* obs, int32_t n,
                            int64_t ld, const uint8_t* labels, const int32_t* boot, int32_t n_trees, int32_t m,
                            int32_t max_depth, int32_t leaf_scale, scoot_node* nodes, int32_t node_cap,
                            int32_t* n_nodes, void* work, int64_t work_bytes, void* stream);
/* Bytes of scratch scoot_rf_train needs for n observations of d features. */
scoot_status scoot_rf_train_work_bytes(int32_t n, int32_t d, int64_t* bytes);

/* ------------------------------------------------------------------ 6. sequential fantasised picks */

/* Bytes of the fantasy state of a GP layout and q picks (host buffer of
 * scoot_fantasy_prepare; about 8 M n^2 bytes). */
scoot_status scoot_fantasy_state_bytes(const scoot_gp_layout* layout, int32_t q, int64_t* bytes);

/* The fp64 state of q sequential fantasised picks, on the host, into h_out
 * (cap bytes, 256-byte aligned when copied to the device): the covariance
 * inputs of the observations (their features, lengthscales, s_f^2, tau^2),
 * alpha = (K + tau^2 I)^{-1} y and L^{-1} (K + tau^2 I = L L^T) in fp64 per
 * objective (Section 4.3), the reference point and the Pareto front of the
 * observations (Section 4.4).  The inputs are those scoot_gp_prepare takes
 * (unwarped states only) plus h_ref [M] and q.  *box_cap (may be NULL)
 * receives the number of boxes the picks may need: the box_cap argument of
 * scoot_fantasy_work_bytes and scoot_suggest_fantasy.  Errors: SCOOT_ENOMEM
 * if cap < scoot_fantasy_state_bytes; SCOOT_EINVAL on bad inputs or a matrix
 * that is not positive definite; SCOOT_EUNSUPPORTED for M outside 2..4 or q
 * outside 1..SCOOT_MAX_Q.  (scoot_round_state_build can write the same state
 * beside the GP blob from one factorisation.) */
scoot_status scoot_fantasy_prepare(const scoot_param* h_space, const scoot_gp_layout* layout,
                                   const uint32_t* h_x_obs, int64_t ld_obs, const float* h_y,
                                   const float* h_lengthscale, const float* h_signal_var,
                                   const float* h_noise_var, const float* h_ref, int32_t q, void* h_out,
                                   int64_t cap, int32_t* box_cap);

/* Bytes of the caller-owned device work buffer scoot_suggest_fantasy needs
 * for a pool of n candidates, q picks and box_cap boxes (about
 * 4 n M (2 + 64 n_rb + q) bytes: moments, whitened covariance rows and
 * downdate factors of every candidate). */
scoot_status scoot_fantasy_work_bytes(const scoot_gp_layout* layout, int64_t n, int32_t q, int32_t box_cap,
                                      int64_t* bytes);

/* q sequential EHVI picks with kriging-believer fantasies (a variant of the
 * parallel suggestion of Section 4.7, whose picks are plain top-k): pick 1 is
 * the EHVI argmax (Eq. 7) over the candidates with mask[i] == 1 (mask may be
 * NULL); after each pick p every objective's value at x_p is fantasised as
 * its posterior mean, the GP is conditioned on it with noise tau^2 (means
 * unchanged, variances lowered by a rank-1 term), the fantasised point joins
 * the Pareto front above the reference point (boxes rebuilt on the device),
 * and the next pick is the EHVI argmax among the candidates not yet picked.
 * Ties go to the lowest index.  state: the GP blob; fant_state: the device
 * copy (256-byte aligned) of scoot_fantasy_prepare's output for the same
 * inputs, with q no larger than the q it was prepared for; box_cap as it
 * returned (or larger).  eps: device base samples [S][M].  work: device
 * buffer of at least scoot_fantasy_work_bytes bytes, 256-byte aligned.
 * Outputs (device): idx int64 [q] and val float [q] (the picks and their
 * EHVI values; -1 and -inf beyond the count), count int32 [1] (fewer than q
 * when the candidates run out); if var_out is not NULL (device [M][n]) it
 * receives the variances after the last downdate for candidates with
 * mask[i] == 1.  Asynchronous on `stream`, with no host synchronisation:
 * the rank-1 terms of every pick are computed on the device in fp64 from
 * fant_state.  Errors found on the device (a fantasy state that does not
 * match the GP layout or a warped GP state: SCOOT_EINVAL; more boxes than
 * box_cap: SCOOT_EUNSUPPORTED) stop the picks and are reported by
 * scoot_ctx_check.  2 <= M <= 4, 1 <= q <= SCOOT_MAX_Q, n < 2^31. */
scoot_status scoot_suggest_fantasy(scoot_ctx* ctx, const scoot_gp_layout* layout, const void* state,
                                   const void* fant_state, int32_t box_cap, const uint32_t* cand, int64_t n,
                                   int64_t ld, const uint8_t* mask, const float* eps, int32_t n_mc, int32_t q,
                                   void* work, int64_t work_bytes, int64_t* idx, float* val, int32_t* count,
                                   float* var_out, void* stream);

/* The same picks over a pool sharded across ranks (one process per GPU,
 * each holding a contiguous share of the candidates and the same GP and
 * fantasy states), as phase calls with one exchange per pick:
 *   scoot_fantasy_begin       compaction of the shard's live candidates, their
 *                             posterior and whitened rows, the observations'
 *                             front and boxes; opens the context's session
 *                             (global index of the shard's candidate 0:
 *                             index_offset; index_offset + n < 2^32);
 *   for j = 0 .. q-1:
 *     scoot_fantasy_local_best   pass j over the shard (the downdate of pick
 *                             j-1, EHVI, the argmax) into rec (device uint64
 *                             [SCOOT_FANT_REC], may be NULL): rec[0] the
 *                             selection key of the shard's best candidate
 *                             (order-preserving bits of its fp32 EHVI value
 *                             << 32 | 0xFFFFFFFF - global index; 0 when the
 *                             shard has no eligible candidate), rec[1 ..] its
 *                             d configuration words, two per element (word
 *                             2k in the low half);
 *     (the caller gathers every rank's record into one device array)
 *     scoot_fantasy_commit    recs: n_rec gathered records (device
 *                             [n_rec][SCOOT_FANT_REC]); the one with the
 *                             largest key is pick j (value descending, global
 *                             index ascending); every rank records it in idx,
 *                             val and count, computes its rank-1 terms from
 *                             the configuration in the record (so no rank
 *                             needs another rank's pool) and rebuilds the
 *                             boxes; the rank holding it excludes it;
 *   scoot_fantasy_end         variances to var_out (may be NULL; the shard's
 *                             [M][n]) and closes the session.
 * Every rank's picks are identical to those of one rank holding the whole
 * pool.  scoot_suggest_fantasy is this sequence on one rank (n_rec = 1).  A
 * context holds one session; no other call on it may come between begin and
 * end (they share its workspace).  All calls are asynchronous on `stream`. */
#define SCOOT_FANT_REC 9
scoot_status scoot_fantasy_begin(scoot_ctx* ctx, const scoot_gp_layout* layout, const void* state,
                                 const void* fant_state, int32_t box_cap, const uint32_t* cand, int64_t n,
                                 int64_t ld, const uint8_t* mask, int64_t index_offset, const float* eps,
                                 int32_t n_mc, int32_t q, void* work, int64_t work_bytes, int64_t* idx, float* val,
                                 int32_t* count, void* stream);
scoot_status scoot_fantasy_local_best(scoot_ctx* ctx, int32_t j, uint64_t* rec, void* stream);
scoot_status scoot_fantasy_commit(scoot_ctx* ctx, int32_t j, const uint64_t* recs, int32_t n_rec, void* stream);
scoot_status scoot_fantasy_end(scoot_ctx* ctx, float* var_out, void* stream);

/* ------------------------------------------------------------------ 7. MACE (Sections 4.5 and 4.7) */

/* Candidates that may survive the pivot stage of scoot_select_pareto (see
 * there). */
#define SCOOT_PARETO_CAP 65536

/* The three acquisition values MACE ranks single-objective candidates by
 * (Section 4.5), from the posterior of objective 0:
 *   UCB = mu + kappa * sigma                  (the UCB equation; kappa is the
 *                                              coefficient beta_t, given by
 *                                              the caller)
 *   PI  = Phi((mu + xi - y_best) / sigma)     (the PI equation; with sigma = 0,
 *                                              1 if mu + xi > y_best, else 0)
 *   EI  as in scoot_acq_ei                    (Eq. 6)
 * acq is [3][lda] (rows UCB, PI, EI; lda >= n); where mask[i] == 0 (mask may
 * be NULL) all three are -inf.  mean/var: objective 0's rows as written by
 * scoot_gp_posterior. */
scoot_status scoot_acq_mace(scoot_ctx* ctx, const float* mean, const float* var, const uint8_t* mask,
                            int64_t n, float y_best, float xi, float kappa, float* acq, int64_t lda,
                            void* stream);

/* scoot_gp_posterior followed by scoot_acq_mace, in one pass (objective 0;
 * y_best is the state's best observed value of objective 0), on the tensor
 * cores or in one fused fp32 kernel as scoot_score_ei. */
scoot_status scoot_score_mace(scoot_ctx* ctx, const scoot_gp_layout* layout, const void* state,
                              const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                              float xi, float kappa, float* acq, int64_t lda, void* stream);

/* Parallel suggestion for one objective (Section 4.7): k candidates drawn at
 * random from the Pareto front of the three rows of acq ([3][lda], each
 * maximised, e.g. as written by scoot_score_mace).  Eligible candidates have
 * mask[i] == 1 (mask may be NULL) and no row NaN or -inf; candidate j
 * dominates i when it is >= in every row and > in one; the front is the
 * eligible candidates no eligible candidate dominates (equal triples are all
 * on it).  The draw gives candidate i the key SplitMix64(seed, i) (output i
 * of the SplitMix64 generator seeded with seed) and takes the k front members
 * with the smallest keys (lower index on equal keys), in that order: a
 * uniformly random k-subset.  Outputs (device): idx (int64 [k], -1 beyond
 * the picks), count (int32 [2]: the number of picks min(k, front size), then
 * the front size) and, if front is not NULL, the first min(front size,
 * front_cap) front members in no particular order.
 * The filter is exact and runs in stages: the front of a strided sample of
 * at most 16384 candidates serves as pivots; every candidate that no pivot
 * dominates is kept, and the kept candidates are filtered against each
 * other.  If more than SCOOT_PARETO_CAP candidates are kept (a front of that
 * size, or pivots that dominate too little), count is {-1, -1}, no pick is
 * made and scoot_ctx_check reports SCOOT_EUNSUPPORTED.
 * 1 <= k <= SCOOT_MAX_Q, n < 2^31. */
scoot_status scoot_select_pareto(scoot_ctx* ctx, const float* acq, int64_t lda, const uint8_t* mask,
                                 int64_t n, int32_t k, uint64_t seed, int64_t* idx, int32_t* count,
                                 int64_t* front, int64_t front_cap, void* stream);

/* scoot_select_topq without a context and without allocating.  The paper
 * has no counterpart: this is a convenience of this library for callers that
 * cannot allocate device memory at selection time (an allocator that forbids
 * allocations while it is active, a process whose device memory is sized up
 * front, or code that cannot create a scoot_ctx because creating one
 * allocates).  Same arguments, semantics and results as scoot_select_topq,
 * on the current CUDA device.  The per-block partial lists live in one
 * fixed 256 KiB device array (32768 keys) that every device which loads the
 * library keeps until the process exits; a call uses at most blocks * q <=
 * 32768 keys, so no pool size overflows it.  The first call on a device
 * looks up the array's device address (make that first call before any
 * stream capture); a lookup that fails returns SCOOT_ECUDA and is tried
 * again by the next call.  An error left pending by the caller's earlier
 * CUDA work is cleared before the launches, so the status reports only this
 * call's own.  All calls share the array: calls that overlap on the GPU
 * (different streams, or different host threads) race and must not be
 * issued; calls ordered on one stream are safe.  Nothing needs clearing
 * between calls: every entry read is written by the same call.  Errors:
 * SCOOT_EUNSUPPORTED for q outside 1..SCOOT_MAX_Q or n >= 2^32,
 * SCOOT_EINVAL for bad pointers or n < 0, SCOOT_ECUDA for runtime failures
 * (there is no context, so no message). */
scoot_status scoot_select_topq_static(const float* acq, const uint8_t* mask, int64_t n, int32_t q,
                                      int64_t* idx, float* val, int32_t* count, void* stream);

/* ------------------------------------------------------------------ measurement probes */

/* Peaks the library's kernels are reported against where no vendor figure
 * applies (the paper has no counterpart; these are measurement aids).
 * scoot_probe_fma: `blocks` blocks of 256 threads, each thread running 16
 * independent fp32 FMA chains for `iters` steps, as scalar FFMAs (packed = 0)
 * or as packed pairs (packed = 1): 2 * 16 * 256 * blocks * iters flops.
 * scoot_probe_gather: `blocks` blocks of 256 threads, each thread taking
 * `steps` dependent steps through a binary tree of n_nodes 8-byte nodes
 * (scoot_node) in shared memory, as a forest walk does (1 <= n_nodes <=
 * 12288): 256 * blocks * steps node visits.  sink: device float [blocks]
 * (receives nothing in practice; it keeps the work live).  Asynchronous. */
scoot_status scoot_probe_fma(scoot_ctx* ctx, int32_t packed, int32_t blocks, int32_t iters, float* sink,
                             void* stream);
scoot_status scoot_probe_gather(scoot_ctx* ctx, int32_t n_nodes, int32_t blocks, int32_t steps, float* sink,
                                void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SCOOT_H */
