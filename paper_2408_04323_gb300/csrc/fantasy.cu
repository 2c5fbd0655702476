// Sequential EHVI picks with kriging-believer fantasies (the parallel-suggestion
// stress variant; the paper's own parallel picks are plain top-k, Section 4.7).
//
// After pick p the value of every objective at x_p is fantasised as its
// posterior mean; conditioning each objective's GP on (x_p, mu(x_p)) with
// noise tau^2 leaves every mean unchanged and lowers every variance by c(x)^2
// with
//   c_j(x) = [k(x, x_p) - v(x).v_p - sum_{l<j} c_l(x) c_l(x_p)] / s_j,
//   s_j    = sqrt(sigma_j^2(x_p) + tau^2),
// where v(x) = L^{-1} k(X, x) are the whitened covariance rows (|v| <= 1, so
// the dot product is well conditioned), sigma_j^2(x_p) is the variance at
// x_p after the previous j fantasies, and l runs over the previous picks.
// The fantasised point joins the Pareto front, the boxes are rebuilt, EHVI
// is recomputed over the pool with the picks excluded, and the next pick is
// its argmax (lowest index on ties).
//
// Everything runs on the device, in stream order, with no host round trip
// (so a whole call can be captured in a CUDA graph):
//   once     compaction of the live candidates; one posterior pass storing
//            mean, variance and V for them by list position (score.cu);
//            fant_init (one block): the observations' front and its boxes;
//   pick j   fant_pass (every live candidate): the downdate of pick j-1, which
//            reads the candidate's rows of V once, then its EHVI over the
//            boxes staged in shared memory, and a per-block argmax;
//            fant_pick (column slabs x objectives): the argmax, then the pick's
//            rank-1 terms in fp64 from the fantasy state: each block takes a
//            slab of columns of L^{-1} and forms its part of v_p = L^{-1} k and
//            of mu(x_p); the last slab of an objective sums the parts and
//            solves for c_l(x_p) and s_j; the last objective adds the
//            fantasised point to the front and rebuilds the boxes.
// GB300 runs fp64 on a narrow pipe (a dependent fp64 operation costs on the
// order of a hundred cycles), so the pick spreads its fp64 work over many
// blocks, keeps dependent chains short (the fantasy factor is kept inverted,
// so its solve is a product), and compares front values as integer keys.
#include <algorithm>
#include <climits>
#include <cmath>
#include <cstring>

#include "device_common.cuh"
#include "internal.h"

namespace {

using namespace scoot_dev;

constexpr int kPassThreads = 256;
constexpr int kCullQueue = 512;        // candidates queued for their exact EHVI per pass block
constexpr int kCullSamplesMax = 256;   // base samples the culling's corners are built from
constexpr int kPickThreads = 256;
constexpr int kPartMax = 2048;   // per-block argmax partials of one pass
constexpr int kPickSlabMax = 32;  // column slabs per objective of the pick's L^{-1} k product

// Column slabs of the pick's product for n observations: about eight columns each.
inline int pick_slabs(int n) { return std::min(kPickSlabMax, std::max(1, (n + 7) / 8)); }

// Control words of one call, in the work buffer.
struct Ctrl {
    uint32_t done;      // 1 once the loop has stopped (no eligible candidate left, or an error)
    uint32_t arrived;   // objectives whose pick terms are final (the last one resets it)
    uint32_t arrived_m[SCOOT_MAX_OBJ];  // row blocks of objective m done (its last one resets it)
    uint32_t passed;    // blocks of the current pass done (the last one resets it)
    int32_t n_boxes;
    int32_t n_front;
    int32_t local_pos;  // list position of this shard's best candidate of the current pass (-1: none)
    uint64_t local_key; // its selection key (global index)
    uint64_t pass_best; // the largest exact selection key found so far in the current pass (culling)
};

struct FantArgs {
    const int32_t* list;          // list position -> candidate index (NULL: identity)
    const unsigned int* n_list;   // live candidates (device; NULL: n)
    int64_t n, ldc;
    const float* mean;            // [M][ldc]
    float* var;                   // [M][ldc]
    const float* V;               // [M][n_pad][ldc]
    float* C;                     // [q][M][ldc] downdate factors c_l of every candidate
    int32_t n_obs, n_pad, d, kernel, q, n_mc, box_cap, front_cap;
    int64_t index_offset;         // global index of this shard's candidate 0 (selection keys, picks)
    const char* gp;               // GP state blob (fp32; feature order)
    int64_t off_fmap, off_ils, off_scal;
    const char* fant;             // fantasy state (fp64; parameter order)
    const uint32_t* cand;
    int64_t ld;
    const float* eps;             // [S][M]
    float* box_lo;                // [box_cap][M]
    float* box_hi;
    double* front;                // [front_cap][M]
    Ctrl* ctrl;
    int64_t* picked_pos;          // [q]
    float* vp;                    // [M][n_pad] v_p of the latest pick (fp32, zero-padded)
    float* cxp;                   // [M][q] c_l(x_p) of the latest pick
    float* inv_s;                 // [M] 1 / s of the latest pick
    double* upick;                // [q][d] features of the picks
    double* vpick;                // [q][M][n] v_p of the picks
    double* wf;                   // [M][q][q] inverse of each objective's fantasy factor (row-major, lower)
    double* part;                 // [M][n_slab][n] each slab's part of v_p
    double* mupart;               // [M][n_slab] each slab's part of mu(x_p)
    double* kpt;                  // [M][q] k(x_p, x_{p_t}) of the earlier picks
    int32_t n_slab, slab_w;       // column slabs of the pick's product and their width
    double* mupick;               // [q][M] fantasised values
    uint64_t* part_key;           // [kPartMax]
    int32_t* part_pos;
    int32_t n_part;               // blocks of a pass
    uint64_t* rec;                // [SCOOT_FANT_REC] this shard's record of the current pass
    uint32_t* pick_words;         // [16] configuration of the latest pick (from the winning record)
    double* fmap64;               // [16][2] offset and scale of each parameter's feature map (feature_map64)
    int64_t* out_idx;             // [q]
    float* out_val;               // [q]
    int32_t* out_count;
    uint32_t* err;
};

__device__ __forceinline__ void keymax(uint64_t& k, int32_t& p, uint64_t k2, int32_t p2) {
    if (k2 > k) {
        k = k2;
        p = p2;
    }
}

// Block-wide maximum of (key, position); valid in thread 0.
__device__ __forceinline__ void block_keymax(uint64_t& k, int32_t& p) {
    __shared__ uint64_t wk[32];
    __shared__ int32_t wp[32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int o = 16; o > 0; o >>= 1) keymax(k, p, __shfl_xor_sync(0xffffffffu, k, o), __shfl_xor_sync(0xffffffffu, p, o));
    if (lane == 0) {
        wk[warp] = k;
        wp[warp] = p;
    }
    __syncthreads();
    if (warp == 0) {
        k = lane < (int)(blockDim.x >> 5) ? wk[lane] : 0ull;
        p = lane < (int)(blockDim.x >> 5) ? wp[lane] : -1;
        for (int o = 16; o > 0; o >>= 1)
            keymax(k, p, __shfl_xor_sync(0xffffffffu, k, o), __shfl_xor_sync(0xffffffffu, p, o));
    }
    __syncthreads();
}

// Sum over a block of kPickThreads threads: the same value, summed in the
// same order, in every thread.
__device__ __forceinline__ double block_sum(double v, double* scratch) {
    static_assert(kPickThreads == 256, "the tree below sums eight warps");
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) scratch[warp] = v;
    __syncthreads();
    const double* w = scratch;
    return ((w[0] + w[1]) + (w[2] + w[3])) + ((w[4] + w[5]) + (w[6] + w[7]));
}

// Sum over warp 0's lanes of v (fixed order), in every lane of warp 0.
__device__ __forceinline__ double warp_sum(double v) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Exclusive prefix over the block (kPickThreads threads) of one flag per
// thread, and the flags' total; every thread calls it.
__device__ __forceinline__ int block_flag_prefix(bool flag, int* warp_tot, int* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const unsigned b = __ballot_sync(0xffffffffu, flag);
    if (lane == 0) warp_tot[warp] = __popc(b);
    __syncthreads();
    int off = 0, tot = 0;
    for (int k = 0; k < nw; ++k) {
        const int c = warp_tot[k];
        off += k < warp ? c : 0;
        tot += c;
    }
    __syncthreads();  // warp_tot may be reused
    *total = tot;
    return off + __popc(b & ((1u << lane) - 1u));
}

// Order-preserving integer key of a double: x < y exactly when key(x) <
// key(y), for values that are not NaN; -0 and +0 share the key of +0.  The
// front and box logic compares these keys on the integer pipes.
__device__ __forceinline__ long long okey(double x) {
    long long b = __double_as_longlong(x);
    if (b == LLONG_MIN) b = 0;  // -0
    return b >= 0 ? b : b ^ LLONG_MAX;
}

__device__ __forceinline__ double okey_value(long long k) { return __longlong_as_double(k >= 0 ? k : k ^ LLONG_MAX); }

__device__ __forceinline__ double matern64(double r, int kernel) {
    if (kernel == SCOOT_MATERN32) {
        const double a = sqrt(3.0) * r;
        return (1.0 + a) * exp(-a);
    }
    const double a = sqrt(5.0) * r;
    return (1.0 + a + a * a / 3.0) * exp(-a);
}

// Offset and scale of parameter c's feature map (fp64): log(lo) and
// 1 / (log(hi) - log(lo)) for integer log-uniform, lo and 1 / (hi - lo) (0
// when hi <= lo) for integer uniform and continuous; computed once per call
// (fant_init), so that a pick's features cost one log at most.
__device__ __forceinline__ void feature_map64(const double* sp, int c, double* fm2) {
    const int kind = (int)sp[c * 4];
    const double lo = sp[c * 4 + 1], hi = sp[c * 4 + 2];
    if (kind == SCOOT_INT_LOG) {
        const double l0 = log(lo);
        fm2[0] = l0;
        fm2[1] = 1.0 / (log(hi) - l0);
    } else {
        fm2[0] = lo;
        fm2[1] = hi > lo ? 1.0 / (hi - lo) : 0.0;
    }
}

// Feature coordinate (fp64) of a stored word of parameter c: log scale for
// integer log-uniform, linear for integer uniform and continuous, the index
// for categoricals (fm2: the offset and scale of feature_map64).  Returns
// false for a word that has no feature.
__device__ __forceinline__ bool feature64(const double* sp, const double* fm2, int c, uint32_t w, double* u) {
    const int kind = (int)sp[c * 4];
    const double v = kind == SCOOT_CONTINUOUS ? (double)__uint_as_float(w) : (double)(int32_t)w;
    if (kind == SCOOT_INT_LOG) {
        if (!(v > 0.0)) return false;
        *u = (log(v) - fm2[2 * c]) * fm2[2 * c + 1];
    } else if (kind == SCOOT_INT_UNIFORM || kind == SCOOT_CONTINUOUS) {
        *u = (v - fm2[2 * c]) * fm2[2 * c + 1];
    } else {
        *u = v;
    }
    return isfinite(*u);
}

// ---------------------------------------------------------------- front and boxes

// Shared-memory need of front_update_and_boxes (bytes).
__host__ __device__ inline size_t boxes_smem(int front_cap, int M, int box_cap) {
    return (size_t)box_cap * 8 + (size_t)front_cap * M * 8 + (size_t)(M - 1) * (front_cap + 1) * 8 +
           (size_t)(front_cap + 1) * 4 + (size_t)(box_cap + 1) * 4 + 64;
}

// One block: optionally adds point z (fp64 of the fp32 fantasised value) to
// the front (if it lies above the reference point and no front point weakly
// dominates it; front points it dominates leave), then decomposes the region
// the front does not dominate into boxes exactly as scoot_boxes_build does:
// columns over the grid of the first M - 1 axes (the reference coordinate and
// the front's, sorted, unique), each open upwards on the last objective from
// max(r_last, the highest last value among front points dominating the
// cell's upper corner), cells merged along the last grid axis while that
// floor repeats.  Boxes in the builder's order.  On a box count beyond
// box_cap the loop stops with a capacity error.
template <int M>
__device__ void front_update_and_boxes(const FantArgs& a, const FantHeader& h, bool add, const double* z,
                                       char* smem) {
    constexpr int G = M - 1;
    const int fcap = a.front_cap;
    // Every value below is an order-preserving key (okey).
    long long* cell = reinterpret_cast<long long*>(smem);           // [box_cap] floor of each grid cell
    long long* F = cell + a.box_cap;                                 // [fcap][M]
    long long* axis = F + (size_t)fcap * M;                          // [G][fcap + 1]
    int32_t* first = reinterpret_cast<int32_t*>(axis + (size_t)G * (fcap + 1));  // [fcap + 1]
    int32_t* rowcnt = first + fcap + 1;                                            // [rows + 1]
    __shared__ int32_t s_nf, s_A[4], s_total, s_ok;
    __shared__ long long s_ref[M];
    const int tid = threadIdx.x;
    if (tid == 0) s_nf = a.ctrl->n_front;
    if (tid < M) s_ref[tid] = okey(h.ref[tid]);
    if (tid < 4) s_A[tid] = 0;
    __syncthreads();
    for (int e = tid; e < s_nf * M; e += blockDim.x) F[e] = okey(a.front[e]);
    __syncthreads();
    __shared__ int s_wt[32];
    if (add) {  // (uniform: every thread takes part in the block-wide steps)
        long long zk[M];
        bool above = true;
#pragma unroll
        for (int m = 0; m < M; ++m) {
            zk[m] = okey(z[m]);
            above &= zk[m] > s_ref[m];
        }
        const int nf0 = s_nf;
        int cov = 0;  // some front point weakly dominates z
        for (int k = tid; k < nf0; k += blockDim.x) {
            bool ge = true;
#pragma unroll
            for (int m = 0; m < M; ++m) ge &= F[k * M + m] >= zk[m];
            cov |= ge;
        }
        const bool covered = __syncthreads_or(cov) != 0;
        if (above && !covered) {
            // Keep, in order, the points z does not dominate (a stable compaction
            // in chunks of the block: a point moves only to a lower position, and
            // every point of a chunk is read before any is written), then z.
            int base = 0;
            for (int c0 = 0; c0 < nf0; c0 += blockDim.x) {
                const int k = c0 + tid;
                long long pt[M];
                bool keep = false;
                if (k < nf0) {
                    bool ge = true, gt = false;
#pragma unroll
                    for (int m = 0; m < M; ++m) {
                        pt[m] = F[k * M + m];
                        ge &= zk[m] >= pt[m];
                        gt |= zk[m] > pt[m];
                    }
                    keep = !(ge && gt);  // not dominated by the fantasy
                }
                int tot;
                const int pos = block_flag_prefix(keep, s_wt, &tot);
                if (keep) {
#pragma unroll
                    for (int m = 0; m < M; ++m) F[(base + pos) * M + m] = pt[m];
                }
                base += tot;
                __syncthreads();
            }
            if (tid == 0) {
                int w = base;
                if (w < fcap) {
                    for (int m = 0; m < M; ++m) F[w * M + m] = zk[m];
                    ++w;
                } else {
                    atomicOr(a.err, SCOOT_DEVERR_CAPACITY);
                }
                s_nf = w;
            }
        }
    }
    __syncthreads();
    const int nf = s_nf;
    for (int e = tid; e < nf * M; e += blockDim.x) a.front[e] = okey_value(F[e]);
    // Axes: {r_j} and the front's coordinates, sorted and unique.  Value t
    // (t = 0 the reference, t = k + 1 front point k) is kept if no earlier t
    // holds the same value; its place is the number of kept values below it.
    for (int j = 0; j < G; ++j) {
        for (int t = tid; t <= nf; t += blockDim.x) {
            const long long v = t == 0 ? s_ref[j] : F[(t - 1) * M + j];
            int f = 1;
            for (int u = 0; u < t && f; ++u) f = (u == 0 ? s_ref[j] : F[(u - 1) * M + j]) != v;
            first[t] = f;
        }
        __syncthreads();
        for (int t = tid; t <= nf; t += blockDim.x) {
            if (!first[t]) continue;
            const long long v = t == 0 ? s_ref[j] : F[(t - 1) * M + j];
            int below = 0;
            for (int u = 0; u <= nf; ++u) below += first[u] && (u == 0 ? s_ref[j] : F[(u - 1) * M + j]) < v;
            axis[j * (fcap + 1) + below] = v;
        }
        int cnt = 0;
        for (int t = tid; t <= nf; t += blockDim.x) cnt += first[t];
        cnt = __reduce_add_sync(0xffffffffu, cnt);
        if ((tid & 31) == 0 && cnt) atomicAdd(&s_A[j], cnt);
        __syncthreads();
    }
    int cells = 1;
    for (int j = 0; j < G; ++j) cells *= s_A[j];
    const int A_last = s_A[G - 1];
    const int rows = cells / A_last;
    if (cells > a.box_cap) {
        if (tid == 0) {
            atomicOr(a.err, SCOOT_DEVERR_CAPACITY);
            a.ctrl->done = 1u;
            a.ctrl->n_boxes = 0;
        }
        return;
    }
    // Floor of every cell (row-major over the grid, the last axis fastest).
    const long long inf = okey(__longlong_as_double(0x7ff0000000000000ll));
    for (int c = tid; c < cells; c += blockDim.x) {
        long long up[G];
        int rest = c;
        for (int j = G - 1; j >= 0; --j) {
            const int kj = rest % s_A[j];
            rest /= s_A[j];
            up[j] = kj + 1 < s_A[j] ? axis[j * (fcap + 1) + kj + 1] : inf;
        }
        long long hh = s_ref[M - 1];
        for (int k = 0; k < nf; ++k) {
            bool dom = true;
            for (int j = 0; j < G; ++j) dom &= F[k * M + j] >= up[j];
            if (dom) hh = max(hh, F[k * M + M - 1]);
        }
        cell[c] = hh;
    }
    __syncthreads();
    // Boxes per row (cells merged while the floor repeats), then their offsets.
    const long long* al = axis + (G - 1) * (fcap + 1);
    if (rows == 1) {
        // One row (two objectives, or one value on every other axis): a box per
        // run of equal floors, the cells in parallel; a cell's box is the number
        // of run starts up to it, less one (a block-wide prefix).
        float lo_pre[G > 1 ? G - 1 : 1], up_pre[G > 1 ? G - 1 : 1];
        for (int j = 0; j < G - 1; ++j) {
            lo_pre[j] = (float)okey_value(axis[j * (fcap + 1)]);
            up_pre[j] = 1 < s_A[j] ? (float)okey_value(axis[j * (fcap + 1) + 1]) : __int_as_float(0x7f800000);
        }
        int base = 0;
        for (int c0 = 0; c0 < A_last; c0 += blockDim.x) {
            const int kk = c0 + tid;
            const bool in = kk < A_last;
            const bool start = in && (kk == 0 || cell[kk] != cell[kk - 1]);
            int tot;
            const int pos = block_flag_prefix(start, s_wt, &tot);
            const int b = base + pos + (start ? 0 : -1);
            if (in && b < a.box_cap) {
                if (start) {
                    for (int j = 0; j < G - 1; ++j) {
                        a.box_lo[b * M + j] = lo_pre[j];
                        a.box_hi[b * M + j] = up_pre[j];
                    }
                    a.box_lo[b * M + G - 1] = (float)okey_value(al[kk]);
                    a.box_lo[b * M + M - 1] = (float)okey_value(cell[kk]);
                    a.box_hi[b * M + M - 1] = __int_as_float(0x7f800000);
                }
                if (kk + 1 == A_last || cell[kk + 1] != cell[kk])  // the run's last cell
                    a.box_hi[b * M + G - 1] = kk + 1 < A_last ? (float)okey_value(al[kk + 1]) : __int_as_float(0x7f800000);
            }
            base += tot;
        }
        if (tid == 0) {
            s_total = base;
            s_ok = base <= a.box_cap;
        }
    } else {
        for (int r = tid; r < rows; r += blockDim.x) {
            int cnt = 1;
            for (int kk = 1; kk < A_last; ++kk) cnt += cell[r * A_last + kk] != cell[r * A_last + kk - 1];
            rowcnt[r + 1] = cnt;
        }
        __syncthreads();
        if (tid == 0) {
            rowcnt[0] = 0;
            for (int r = 0; r < rows; ++r) rowcnt[r + 1] += rowcnt[r];
            s_total = rowcnt[rows];
            s_ok = s_total <= a.box_cap;
        }
        __syncthreads();
        for (int r = tid; r < rows && s_ok; r += blockDim.x) {
            float lo_pre[G > 1 ? G - 1 : 1], up_pre[G > 1 ? G - 1 : 1];
            int rest = r;
            for (int j = G - 2; j >= 0; --j) {
                const int kj = rest % s_A[j];
                rest /= s_A[j];
                lo_pre[j] = (float)okey_value(axis[j * (fcap + 1) + kj]);
                up_pre[j] = kj + 1 < s_A[j] ? (float)okey_value(axis[j * (fcap + 1) + kj + 1]) : __int_as_float(0x7f800000);
            }
            int b = rowcnt[r] - 1;
            for (int kk = 0; kk < A_last; ++kk) {
                const long long fl = cell[r * A_last + kk];
                if (kk == 0 || fl != cell[r * A_last + kk - 1]) {
                    ++b;
                    for (int j = 0; j < G - 1; ++j) {
                        a.box_lo[b * M + j] = lo_pre[j];
                        a.box_hi[b * M + j] = up_pre[j];
                    }
                    a.box_lo[b * M + G - 1] = (float)okey_value(al[kk]);
                    a.box_lo[b * M + M - 1] = (float)okey_value(fl);
                    a.box_hi[b * M + M - 1] = __int_as_float(0x7f800000);
                }
                a.box_hi[b * M + G - 1] = kk + 1 < A_last ? (float)okey_value(al[kk + 1]) : __int_as_float(0x7f800000);
            }
        }
    }
    __syncthreads();
    if (tid == 0) {
        a.ctrl->n_front = nf;
        if (s_ok) {
            a.ctrl->n_boxes = s_total;
        } else {
            atomicOr(a.err, SCOOT_DEVERR_CAPACITY);
            a.ctrl->done = 1u;
            a.ctrl->n_boxes = 0;
        }
    }
}

// ---------------------------------------------------------------- records

// The last block of a pass to finish reduces the per-block partials to this
// shard's record: the selection key of its best candidate (global index)
// and that candidate's d configuration words, two per 64-bit word (word 2k
// in the low half); key 0 when the shard has no eligible candidate left.
__device__ void pass_record(const FantArgs& a) {
    __shared__ int s_last;
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_last = atomicAdd(&a.ctrl->passed, 1u) == gridDim.x - 1;
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    uint64_t best = 0ull;
    int32_t pos = -1;
    for (int k = threadIdx.x; k < (int)gridDim.x; k += blockDim.x)
        keymax(best, pos, __ldcg(a.part_key + k), __ldcg(a.part_pos + k));
    block_keymax(best, pos);
    if (threadIdx.x == 0) {
        a.ctrl->passed = 0u;
        a.ctrl->pass_best = 0ull;  // for the next pass
        a.ctrl->local_key = best;
        a.ctrl->local_pos = best != 0ull ? pos : -1;
        a.rec[0] = best;
    }
    if (threadIdx.x < (SCOOT_FANT_REC - 1)) {
        uint64_t w = 0ull;
        if (best != 0ull) {
            const int64_t i = a.list ? (int64_t)a.list[pos] : (int64_t)pos;
            const int c0 = 2 * threadIdx.x, c1 = c0 + 1;
            const uint32_t lo = c0 < a.d ? __ldg(a.cand + (int64_t)c0 * a.ld + i) : 0u;
            const uint32_t hi = c1 < a.d ? __ldg(a.cand + (int64_t)c1 * a.ld + i) : 0u;
            w = (uint64_t)lo | ((uint64_t)hi << 32);
        }
        a.rec[1 + threadIdx.x] = w;
    }
}

// ---------------------------------------------------------------- kernels

// One block: checks the fantasy state against the call, resets the control
// words and outputs, and decomposes the observations' front into boxes.
template <int M>
__global__ void __launch_bounds__(kPickThreads) fant_init(const __grid_constant__ FantArgs a) {
    extern __shared__ __align__(16) char smem[];
    const FantHeader& h = *reinterpret_cast<const FantHeader*>(a.fant);
    const float* gscal = reinterpret_cast<const float*>(a.gp + a.off_scal);
    __shared__ int ok;
    if (threadIdx.x == 0) {
        ok = h.magic == kFantMagic && h.n == a.n_obs && h.d == a.d && h.M == M && h.q >= a.q &&
             h.kernel == a.kernel && h.front0 >= 0 && h.front0 <= a.n_obs;
        for (int m = 0; m < M; ++m) ok &= gscal[m * 4 + 3] == 0.0f;  // an unwarped GP state
        a.ctrl->done = ok ? 0u : 1u;
        a.ctrl->arrived = 0u;
        for (int m = 0; m < SCOOT_MAX_OBJ; ++m) a.ctrl->arrived_m[m] = 0u;
        a.ctrl->passed = 0u;
        a.ctrl->pass_best = 0ull;
        a.ctrl->local_key = 0ull;
        a.ctrl->local_pos = -1;
        a.ctrl->n_boxes = 0;
        a.ctrl->n_front = ok ? h.front0 : 0;
        *a.out_count = 0;
        if (!ok) atomicOr(a.err, SCOOT_DEVERR_VALUE);
    }
    for (int j = threadIdx.x; j < a.q; j += blockDim.x) {
        a.out_idx[j] = -1;
        a.out_val[j] = -INFINITY;
    }
    __syncthreads();
    if (!ok) return;
    const double* f0 = reinterpret_cast<const double*>(a.fant + h.off_front);
    for (int e = threadIdx.x; e < h.front0 * M; e += blockDim.x) a.front[e] = f0[e];
    if (threadIdx.x < a.d)
        feature_map64(reinterpret_cast<const double*>(a.fant + h.off_space), threadIdx.x, a.fmap64 + 2 * threadIdx.x);
    __syncthreads();
    front_update_and_boxes<M>(a, h, false, nullptr, smem);
}

// Pick j's pass over the live candidates: for j > 0 the downdate of pick
// j - 1, then EHVI over the current boxes with the picks excluded, and each
// block's best (key, list position).
template <int M>
__global__ void __launch_bounds__(kPassThreads, M == 2 ? 4 : 1) fant_pass(const __grid_constant__ FantArgs a, int j) {
    // Two objectives fit 64 registers without spills: four blocks (32 warps)
    // per SM keep more rows of V in flight.
    if (*(volatile const uint32_t*)&a.ctrl->done) {
        if (threadIdx.x == 0) a.part_key[blockIdx.x] = 0ull;
        return;
    }
    extern __shared__ __align__(16) float sm[];
    const int nb = a.ctrl->n_boxes;
    float4* blo = reinterpret_cast<float4*>(sm);
    float4* bhi = blo + nb;
    float4* epsv = bhi + nb;
    int64_t* pk = reinterpret_cast<int64_t*>(epsv + a.n_mc);  // [q] list positions of the picks
    float* vps = reinterpret_cast<float*>(pk + ((a.q + 1) & ~1));  // [M][n_pad] (16-byte aligned)
    float* cxs = vps + M * a.n_pad;                           // [M][q]
    float* ins = cxs + M * a.q;                               // [M]
    float* ups = ins + M;                                     // [d] features of the latest pick (feature order)
    const float4* fm = reinterpret_cast<const float4*>(a.gp + a.off_fmap);
    const float* gils = reinterpret_cast<const float*>(a.gp + a.off_ils);
    const float* gscal = reinterpret_cast<const float*>(a.gp + a.off_scal);
    stage_boxes(a.box_lo, a.box_hi, nb, a.eps, a.n_mc, M, blo, bhi, epsv);
    const int l = j - 1;  // the downdate of this pass
    if (l >= 0) {
        for (int e = threadIdx.x; e < M * a.n_pad; e += blockDim.x) vps[e] = a.vp[e];
        for (int e = threadIdx.x; e < M * a.q; e += blockDim.x) cxs[e] = a.cxp[e];
        if (threadIdx.x < M) ins[threadIdx.x] = a.inv_s[threadIdx.x];
        for (int c = threadIdx.x; c < a.d; c += blockDim.x) {
            const float4 f = fm[c];
            ups[c] = feature_of(a.pick_words[(int)f.w], (int)f.x, f.y, f.z);
        }
    }
    for (int e = threadIdx.x; e < j; e += blockDim.x) pk[e] = a.picked_pos[e];
    __syncthreads();
    const bool fast = boxes_fast(blo, bhi, nb, M);
    if (fast) {
        stage_boxes_sat(a.box_lo, a.box_hi, nb, M, blo);
        __syncthreads();
    }
    const int64_t n_live = a.n_list ? (int64_t)*a.n_list : a.n;
    uint64_t best = 0ull;
    int32_t best_pos = -1;
    const float inv_mc = 1.0f / (float)a.n_mc;
    // The downdate of the candidate at list position pos (pick j - 1's rank-1
    // term, stored), and its variances.
    auto downdate = [&](int64_t pos, int64_t i, float* vr) {
        if (l >= 0) {
            float r2[M];
#pragma unroll
            for (int m = 0; m < M; ++m) r2[m] = 0.0f;
            for (int c = 0; c < a.d; ++c) {
                const float4 f = fm[c];
                const int kind = (int)f.x;
                const float ux = feature_of(__ldg(a.cand + (int64_t)f.w * a.ld + i), kind, f.y, f.z);
                const float up = ups[c];
#pragma unroll
                for (int m = 0; m < M; ++m) {
                    const float s = gils[m * a.d + c];
                    if (kind == SCOOT_CATEGORICAL) {
                        r2[m] += ux != up ? s : 0.0f;
                    } else {
                        const float t = (ux - up) * s;
                        r2[m] = fmaf(t, t, r2[m]);
                    }
                }
            }
#pragma unroll
            for (int m = 0; m < M; ++m) {
                const float k = gscal[m * 4] * matern(sqrtf(r2[m]), a.kernel);
                // v(x) . v_p over float4 groups of four rows (16-byte loads;
                // rows past n_obs are zero on both sides).
                const float4* vrow = reinterpret_cast<const float4*>(a.V) + vtile_index(pos, m, 0, M, a.n_pad / 4);
                const float4* vpm = reinterpret_cast<const float4*>(vps + m * a.n_pad);
                const int groups = (a.n_obs + 3) / 4;
                float d0 = 0.0f, d1 = 0.0f, d2 = 0.0f, d3 = 0.0f;
#pragma unroll 8
                for (int g = 0; g < groups; ++g) {
                    const float4 v = __ldcs(vrow + 32 * g);
                    const float4 w = vpm[g];
                    d0 = fmaf(v.x, w.x, d0);
                    d1 = fmaf(v.y, w.y, d1);
                    d2 = fmaf(v.z, w.z, d2);
                    d3 = fmaf(v.w, w.w, d3);
                }
                float cc = 0.0f;
                for (int t = 0; t < l; ++t) cc = fmaf(a.C[((int64_t)t * M + m) * a.ldc + pos], cxs[m * a.q + t], cc);
                const float c = (k - ((d0 + d1) + (d2 + d3)) - cc) * ins[m];
                if (l < a.q - 2) a.C[((int64_t)l * M + m) * a.ldc + pos] = c;  // read by later downdates
                float* vv = a.var + (int64_t)m * a.ldc + pos;
                vr[m] = fmaxf(*vv - c * c, 0.0f);
                *vv = vr[m];
            }
        } else {
#pragma unroll
            for (int m = 0; m < M; ++m) vr[m] = a.var[(int64_t)m * a.ldc + pos];
        }
    };
    auto exact = [&](const float* mu, const float* sd) -> float {
        if constexpr (M <= 3)  // (the saturated form takes two or three objectives)
            return fast ? ehvi_partial_sat<M>(mu, sd, blo, nb, epsv, a.n_mc, 0, 1) * inv_mc
                        : ehvi_value<M>(mu, sd, blo, bhi, nb, epsv, a.n_mc);
        else
            return ehvi_value<M>(mu, sd, blo, bhi, nb, epsv, a.n_mc);
    };
    const bool cull = fast && a.n_mc >= 16 && a.n_mc % 8 == 0 && a.n_mc <= kCullSamplesMax;
    if (!cull) {
        for (int64_t pos = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; pos < n_live;
             pos += (int64_t)gridDim.x * blockDim.x) {
            const int64_t i = a.list ? (int64_t)a.list[pos] : pos;
            float vr[M];
            downdate(pos, i, vr);
            bool taken = false;
            for (int t = 0; t < j; ++t) taken |= pk[t] == pos;
            if (taken) continue;
            float mu[M], sd[M];
#pragma unroll
            for (int m = 0; m < M; ++m) {
                mu[m] = a.mean[(int64_t)m * a.ldc + pos];
                sd[m] = sqrtf(fmaxf(vr[m], 0.0f));
            }
            const float v = exact(mu, sd);
            if (!(v != v) && v != -INFINITY)
                keymax(best, best_pos, make_key(v, (uint32_t)(a.index_offset + i)), (int32_t)pos);
        }
    } else if constexpr (M <= 3) {
        // Culling.  The samples, in 8-sample groups by rank of their first
        // objective, give corners (the group's largest value per objective);
        // the HVI is monotone in each objective (and its computed form too:
        // every operation is monotone), so the group size times the HVI at
        // the corner bounds the group's HVI sum, and the corners' sum bounds
        // the EHVI.  A candidate whose bound's selection key (the bound
        // raised by 2^-16 against the sums' roundings) is below the largest
        // exact key found so far (this block's or any block's) cannot be the
        // pass's argmax and skips its EHVI; the others queue in shared memory
        // and are evaluated a block-full at a time, so a warp's lanes all have
        // work.
        const int ng = a.n_mc / 8;
        float4* cornv = reinterpret_cast<float4*>(reinterpret_cast<uintptr_t>(ups + a.d + 3) & ~(uintptr_t)15);  // [ng]
        int* rk = reinterpret_cast<int*>(cornv + ng);                   // [n_mc]
        float* qmu = reinterpret_cast<float*>(rk + a.n_mc);              // [M][kCullQueue]
        float* qsd = qmu + M * kCullQueue;                               // [M][kCullQueue]
        int32_t* qpos = reinterpret_cast<int32_t*>(qsd + M * kCullQueue); // [kCullQueue]
        uint32_t* qidx = reinterpret_cast<uint32_t*>(qpos + kCullQueue);  // [kCullQueue]
        __shared__ unsigned long long s_best;
        __shared__ int s_qn;
        for (int s = threadIdx.x; s < a.n_mc; s += blockDim.x) {
            const float e0 = epsv[s].x;
            int r = 0;
            for (int u = 0; u < a.n_mc; ++u) r += epsv[u].x < e0 || (epsv[u].x == e0 && u < s);
            rk[s] = r;
        }
        if (threadIdx.x == 0) {
            s_best = 0ull;
            s_qn = 0;
        }
        __syncthreads();
        for (int g = threadIdx.x; g < ng; g += blockDim.x) {
            float4 c = make_float4(-INFINITY, -INFINITY, -INFINITY, 0.0f);
            for (int s = 0; s < a.n_mc; ++s)
                if (rk[s] / 8 == g) {
                    const float4 e = epsv[s];
                    c.x = fmaxf(c.x, e.x);
                    c.y = fmaxf(c.y, e.y);
                    c.z = fmaxf(c.z, e.z);
                }
            if (M < 3) c.z = 0.0f;
            cornv[g] = c;
        }
        __syncthreads();
        const int64_t first = (int64_t)blockIdx.x * blockDim.x;
        const int64_t stride = (int64_t)gridDim.x * blockDim.x;
        const int64_t rounds = first < n_live ? (n_live - first + stride - 1) / stride : 0;  // block-uniform
        unsigned long long gb = 0ull;
        for (int64_t rd = 0; rd < rounds; ++rd) {
            const int64_t pos = first + rd * stride + threadIdx.x;
            const bool valid = pos < n_live;
            const unsigned long long gb_next = *(volatile const unsigned long long*)&a.ctrl->pass_best;
            if (valid) {
                const int64_t i = a.list ? (int64_t)a.list[pos] : pos;
                float vr[M];
                downdate(pos, i, vr);
                bool taken = false;
                for (int t = 0; t < j; ++t) taken |= pk[t] == pos;
                if (!taken) {
                    float mu[M], sd[M];
#pragma unroll
                    for (int m = 0; m < M; ++m) {
                        mu[m] = a.mean[(int64_t)m * a.ldc + pos];
                        sd[m] = sqrtf(fmaxf(vr[m], 0.0f));
                    }
                    const uint32_t gi = (uint32_t)(a.index_offset + i);
                    const float ub = ehvi_partial_sat<M>(mu, sd, blo, nb, cornv, ng, 0, 1) * (8.0f * inv_mc);
                    const unsigned long long th = max(s_best, gb);
                    if (ub != ub || make_key(ub * (1.0f + 1.0f / 65536.0f), gi) > th) {
                        const int slot = atomicAdd(&s_qn, 1);
#pragma unroll
                        for (int m = 0; m < M; ++m) {
                            qmu[m * kCullQueue + slot] = mu[m];
                            qsd[m * kCullQueue + slot] = sd[m];
                        }
                        qpos[slot] = (int32_t)pos;
                        qidx[slot] = gi;
                    }
                }
            }
            gb = max(gb, gb_next);
            __syncthreads();
            const int qn = s_qn;
            if (qn >= (int)blockDim.x || rd + 1 == rounds) {
                for (int e = threadIdx.x; e < qn; e += blockDim.x) {
                    float mu[M], sd[M];
#pragma unroll
                    for (int m = 0; m < M; ++m) {
                        mu[m] = qmu[m * kCullQueue + e];
                        sd[m] = qsd[m * kCullQueue + e];
                    }
                    const float v = exact(mu, sd);
                    if (!(v != v) && v != -INFINITY) {
                        const uint64_t key = make_key(v, qidx[e]);
                        keymax(best, best_pos, key, qpos[e]);
                        atomicMax(&s_best, (unsigned long long)key);
                    }
                }
                __syncthreads();
                if (threadIdx.x == 0) {
                    s_qn = 0;
                    atomicMax((unsigned long long*)&a.ctrl->pass_best, s_best);
                }
                __syncthreads();
            }
        }
    }
    block_keymax(best, best_pos);
    if (threadIdx.x == 0) {
        a.part_key[blockIdx.x] = best;
        a.part_pos[blockIdx.x] = best_pos;
    }
    pass_record(a);
}

// Pick j, on a grid of n_slab x M blocks.  Every block reduces the shards'
// records to the winner; block (0, 0) records the pick.  Block (b, m) then
// evaluates k(X_c, x_p) of objective m for the columns c of slab b, and
// forms that slab's part of v_p = L^{-1} k (sum over its columns, every row
// below them) and of mu(x_p) = alpha . k, plus k(x_p, x_{p_t}) for the
// earlier picks t = b, b + n_slab, ...  The last slab of objective m to
// finish sums the parts (in slab order) and completes that objective's
// terms: |v_p|^2, v_p . v_{p_t}, c(x_p) = W (k(x_p, x_{p_t}) - v_p . v_{p_t})
// with W the inverse of the fantasy factor (row t: c_l(x_{p_t}) for l < t,
// s_t on the diagonal), s_j, the new row of W, and the fp32 copies the next
// pass reads.  The last objective to finish adds the fantasised point to
// the front and rebuilds the boxes.
template <int M>
__global__ void __launch_bounds__(kPickThreads) fant_pick(const __grid_constant__ FantArgs a, int j,
                                                          const uint64_t* recs, int n_rec) {
    extern __shared__ __align__(16) char smem[];
    if (*(volatile const uint32_t*)&a.ctrl->done) return;
    const FantHeader& h = *reinterpret_cast<const FantHeader*>(a.fant);
    const int tid = threadIdx.x, b = blockIdx.x, m = blockIdx.y, B = gridDim.x;
    // The winning record: the largest selection key over the shards.
    __shared__ uint64_t s_best;
    __shared__ int32_t s_win;
    __shared__ uint32_t s_words[16];
    if (tid == 0) {
        uint64_t best = 0ull;
        int win = -1;
        for (int k = 0; k < n_rec; ++k) {
            const uint64_t key = __ldcg(recs + (size_t)k * SCOOT_FANT_REC);
            if (key > best) {
                best = key;
                win = k;
            }
        }
        s_best = best;
        s_win = win;
    }
    __syncthreads();
    const uint64_t best = s_best;
    const bool lead = b == 0 && m == 0;
    if (best == 0ull) {  // no eligible candidate left on any shard: the picks end here
        if (lead && tid == 0) a.ctrl->done = 1u;
        return;
    }
    if (tid < 16) {
        const uint64_t w = __ldcg(recs + (size_t)s_win * SCOOT_FANT_REC + 1 + tid / 2);
        s_words[tid] = (tid & 1) ? (uint32_t)(w >> 32) : (uint32_t)w;
    }
    __syncthreads();
    const int64_t p = key_index(best);
    if (lead && tid == 0) {
        const bool owner = a.ctrl->local_key == best;  // this shard holds the pick
        a.out_idx[j] = p;
        a.out_val[j] = key_value(best);
        *a.out_count = j + 1;
        a.picked_pos[j] = owner ? a.ctrl->local_pos : -1;
    }
    if (lead && tid < a.d) a.pick_words[tid] = s_words[tid];
    if (j + 1 >= a.q) return;  // no later pick needs this one's fantasy
    const int n = a.n_obs, d = a.d, q = a.q;
    const double* sp = reinterpret_cast<const double*>(a.fant + h.off_space);
    const double* uo = reinterpret_cast<const double*>(a.fant + h.off_u);
    const double* ell = reinterpret_cast<const double*>(a.fant + h.off_ell) + (size_t)m * d;
    const double* alpha = reinterpret_cast<const double*>(a.fant + h.off_alpha) + (size_t)m * n;
    const double* Li = reinterpret_cast<const double*>(a.fant + h.off_linv) + (size_t)m * n * n;
    const double sf2 = h.sf2[m], tau2 = h.tau2[m];
    double* u = reinterpret_cast<double*>(smem);     // [16] features of the pick
    double* il = u + 16;                              // [16] 1/l (ordinal) or 1/l^2 (categorical)
    double* ks = il + 16;                             // [slab_w] k(X_c, x_p) of this slab's columns
    __shared__ int s_bad, s_last, s_cat[16];
    if (tid == 0) s_bad = 0;
    __syncthreads();
    if (tid < d) {  // the pick's features (one thread each) ...
        double x = 0.0;
        if (!feature64(sp, a.fmap64, tid, s_words[tid], &x)) s_bad = 1;
        u[tid] = x;
        if (lead) a.upick[(size_t)j * d + tid] = x;
    } else if (tid >= 32 && tid < 32 + d) {  // ... and, in another warp, the length scales
        const int c = tid - 32;
        const bool cat = (int)sp[c * 4] == SCOOT_CATEGORICAL;
        s_cat[c] = cat;
        il[c] = cat ? 1.0 / (ell[c] * ell[c]) : 1.0 / ell[c];
    }
    __syncthreads();
    if (s_bad) {
        if (tid == 0) {
            atomicOr(a.err, SCOOT_DEVERR_VALUE);
            a.ctrl->done = 1u;
        }
        return;
    }
    // k(x_p, x), fp64: ordinal coordinates times 1/l, categorical mismatches 1/l^2.
    auto cov = [&](const double* ub) {
        double r2 = 0.0;
        for (int c = 0; c < d; ++c) {
            if (s_cat[c]) {
                r2 += u[c] != ub[c] ? il[c] : 0.0;
            } else {
                const double t = (u[c] - ub[c]) * il[c];
                r2 = fma(t, t, r2);
            }
        }
        return sf2 * matern64(sqrt(r2), a.kernel);
    };
    const int w = a.slab_w, c0 = b * w, c1 = min(n, c0 + w);
    for (int c = c0 + tid; c < c1; c += blockDim.x) ks[c - c0] = cov(uo + (size_t)c * d);
    for (int t = b + B * (int)(blockDim.x - 1 - tid); t < j; t += B * (int)blockDim.x)  // top threads
        a.kpt[(size_t)m * q + t] = cov(a.upick + (size_t)t * d);
    __syncthreads();
    if (tid < 32) {
        double s = 0.0;
        for (int c = c0 + tid; c < c1; c += 32) s = fma(alpha[c], ks[c - c0], s);
        s = warp_sum(s);
        if (tid == 0) a.mupart[(size_t)m * B + b] = s;
    }
    // Rows i >= c0 of this slab's part: sum over its columns c <= i of L^{-1}[i][c] k_c
    // (L^{-1} column-major: the threads of a warp read consecutive rows of a column).
    double* part = a.part + ((size_t)m * B + b) * n;
    for (int i = c0 + tid; i < n; i += blockDim.x) {
        const int ce = min(c1, i + 1);
        double s0 = 0.0, s1 = 0.0;
        int c = c0;
        for (; c + 1 < ce; c += 2) {
            s0 = fma(Li[(size_t)c * n + i], ks[c - c0], s0);
            s1 = fma(Li[(size_t)(c + 1) * n + i], ks[c + 1 - c0], s1);
        }
        if (c < ce) s0 = fma(Li[(size_t)c * n + i], ks[c - c0], s0);
        part[i] = s0 + s1;
    }
    // The last slab of objective m completes its terms.
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(&a.ctrl->arrived_m[m], 1u) == (unsigned)(B - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (tid == 0) a.ctrl->arrived_m[m] = 0u;
    double* vv = reinterpret_cast<double*>(smem);  // [n] v_p
    double* D = vv + n;                            // [q] v_p . v_{p_t}
    double* bq = D + q;                            // [q] k(x_p, x_{p_t}), then minus v_p . v_{p_t}
    double* cq = bq + q;                           // [q] c_t(x_p)
    double* red = cq + q;                          // [32]
    double* red2 = red + 32;                       // [32]
    double* Ws = red2 + 32;                        // [j][q] rows of W of the earlier picks
    // The phase's global reads go out together (an in-order pipe would
    // otherwise wait for each load before issuing the next): W's rows and
    // k(x_p, x_{p_t}) into shared memory, each thread's slab parts into registers.
    const double* W = a.wf + (size_t)m * q * q;
    for (int e = tid; e < j * q; e += blockDim.x) Ws[e] = W[e];
    for (int t = tid; t < j; t += blockDim.x) bq[t] = __ldcg(a.kpt + (size_t)m * q + t);
    const double* pm = a.part + (size_t)m * B * n;
    double* vrow = a.vpick + ((size_t)j * M + m) * n;
    double vv_part = 0.0;
    for (int i = tid; i < n; i += blockDim.x) {
        const int nb = min(B, i / w + 1);  // the slabs with c0 <= i, summed in slab order, k mod 4 apart
        double pv[kPickSlabMax];
#pragma unroll
        for (int k = 0; k < kPickSlabMax; ++k) pv[k] = __ldcg(pm + (size_t)min(k, nb - 1) * n + i);
        double sk[4] = {0.0, 0.0, 0.0, 0.0};
#pragma unroll
        for (int k = 0; k < kPickSlabMax; ++k) sk[k & 3] += k < nb ? pv[k] : 0.0;
        const double v = (sk[0] + sk[1]) + (sk[2] + sk[3]);
        vv[i] = v;
        vrow[i] = v;
        a.vp[m * a.n_pad + i] = (float)v;
        vv_part = fma(v, v, vv_part);
    }
    for (int i = n + tid; i < a.n_pad; i += blockDim.x) a.vp[m * a.n_pad + i] = 0.0f;
    if (tid < 32) {
        double s = 0.0;
        for (int k = tid; k < B; k += 32) s += __ldcg(a.mupart + (size_t)m * B + k);
        s = warp_sum(s);
        if (tid == 0) a.mupick[(size_t)j * M + m] = s;
    }
    const double vnorm = block_sum(vv_part, red);  // (its barriers also publish vv, Ws and bq)
    {  // v_p . v_{p_t}: a warp per two earlier picks, eight rows per lane loaded before use
        const int lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
        for (int t = warp; t < j; t += 2 * nw) {
            const int t2 = t + nw < j ? t + nw : t;
            const double* va = a.vpick + ((size_t)t * M + m) * n;
            const double* vb = a.vpick + ((size_t)t2 * M + m) * n;
            double sa = 0.0, sb = 0.0;
            for (int i0 = lane; i0 < n; i0 += 32 * 8) {
                double xa[8], xb[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int i = min(i0 + 32 * u, n - 1);
                    xa[u] = va[i];
                    xb[u] = vb[i];
                }
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    if (i0 + 32 * u < n) {
                        sa = fma(vv[i0 + 32 * u], xa[u], sa);
                        sb = fma(vv[i0 + 32 * u], xb[u], sb);
                    }
            }
            for (int o = 16; o > 0; o >>= 1) {
                sa += __shfl_xor_sync(0xffffffffu, sa, o);
                sb += __shfl_xor_sync(0xffffffffu, sb, o);
            }
            if (lane == 0) {
                D[t] = sa;
                D[t2] = sb;
            }
        }
    }
    __syncthreads();
    for (int t = tid; t < j; t += blockDim.x) bq[t] -= D[t];
    __syncthreads();
    // c(x_p) = W b: row t of W holds t + 1 entries.
    double csq = 0.0;
    for (int t = tid; t < j; t += blockDim.x) {
        const double* wt = Ws + (size_t)t * q;
        double s0 = 0.0, s1 = 0.0, s2 = 0.0, s3 = 0.0;
        int k = 0;
        for (; k + 3 <= t; k += 4) {
            s0 = fma(wt[k], bq[k], s0);
            s1 = fma(wt[k + 1], bq[k + 1], s1);
            s2 = fma(wt[k + 2], bq[k + 2], s2);
            s3 = fma(wt[k + 3], bq[k + 3], s3);
        }
        for (; k <= t; ++k) s0 = fma(wt[k], bq[k], s0);
        const double c = (s0 + s1) + (s2 + s3);
        cq[t] = c;
        csq = fma(c, c, csq);
    }
    const double csum = block_sum(csq, red2);  // (its barriers also publish cq)
    // s_j^2 = sigma^2(x_p) - sum_t c_t(x_p)^2 + tau^2; 1/s_j from one reciprocal square root.
    const double x = fmax(sf2 - vnorm - csum, 0.0) + tau2;
    const double inv = x > 0.0 ? rsqrt(x) : 0.0;
    if (tid == 0) a.inv_s[m] = (float)inv;
    // Row j of W: -(1/s_j) sum_{k=t}^{j-1} c_k W[k][t] for t < j, 1/s_j on the diagonal.
    double* wj = a.wf + ((size_t)m * q + j) * q;
    for (int t = tid; t <= j; t += blockDim.x) {
        if (t == j) {
            wj[t] = inv;
            continue;
        }
        double s0 = 0.0, s1 = 0.0;
        int k = t;
        for (; k + 1 < j; k += 2) {
            s0 = fma(cq[k], Ws[(size_t)k * q + t], s0);
            s1 = fma(cq[k + 1], Ws[(size_t)(k + 1) * q + t], s1);
        }
        if (k < j) s0 = fma(cq[k], Ws[(size_t)k * q + t], s0);
        wj[t] = -inv * (s0 + s1);
    }
    for (int t = tid; t < q; t += blockDim.x) a.cxp[m * q + t] = t < j ? (float)cq[t] : 0.0f;
    // The last objective adds the fantasised point and rebuilds the boxes.
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(&a.ctrl->arrived, 1u) == (unsigned)(M - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (tid == 0) a.ctrl->arrived = 0u;
    double z[M];
#pragma unroll
    for (int k = 0; k < M; ++k) z[k] = (double)(float)__ldcg(a.mupick + (size_t)j * M + k);
    front_update_and_boxes<M>(a, h, true, z, smem);
}

__global__ void __launch_bounds__(kPassThreads)
scatter_var(const int32_t* list, const unsigned int* n_list, int64_t n, int64_t ldc, int M, const float* var,
            float* out, int64_t ldo) {
    const int64_t n_live = n_list ? (int64_t)*n_list : n;
    for (int64_t pos = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; pos < n_live;
         pos += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = list ? (int64_t)list[pos] : pos;
        for (int m = 0; m < M; ++m) out[(int64_t)m * ldo + i] = var[(int64_t)m * ldc + pos];
    }
}

// ---------------------------------------------------------------- work buffer

struct WorkLayout {
    int64_t mean, var, V, C, ctrl, picked, vp, cxp, inv_s, upick, vpick, wf, part, mupart, kpt, mupick, front,
        box_lo, box_hi, part_key, part_pos, rec, words, fmap64, tcb, tcb_bytes, bytes;
};

int64_t up256(int64_t x) { return (x + 255) / 256 * 256; }

WorkLayout work_layout(const scoot_gp_layout* L, int64_t n, int q, int box_cap) {
    const int64_t M = L->n_obj, n_pad = (int64_t)L->n_rb * 64, no = L->n, d = L->d;
    const int64_t fcap = no + q;
    WorkLayout w;
    int64_t o = 0;
    w.mean = o;     o = up256(o + M * n * 4);
    w.var = o;      o = up256(o + M * n * 4);
    w.V = o;        o = up256(o + M * n_pad * ((n + 31) / 32 * 32) * 4);  // tiled by 32 candidates
    w.C = o;        o = up256(o + (int64_t)std::max(q - 2, 1) * M * n * 4);
    w.ctrl = o;     o = up256(o + (int64_t)sizeof(Ctrl));
    w.picked = o;   o = up256(o + (int64_t)q * 8);
    w.vp = o;       o = up256(o + M * n_pad * 4);
    w.cxp = o;      o = up256(o + M * q * 4);
    w.inv_s = o;    o = up256(o + M * 4);
    w.upick = o;    o = up256(o + (int64_t)q * d * 8);
    w.vpick = o;    o = up256(o + (int64_t)q * M * no * 8);
    w.wf = o;       o = up256(o + M * q * q * 8);
    w.part = o;     o = up256(o + M * pick_slabs((int)no) * no * 8);
    w.mupart = o;   o = up256(o + M * pick_slabs((int)no) * 8);
    w.kpt = o;      o = up256(o + M * q * 8);
    w.mupick = o;   o = up256(o + (int64_t)q * M * 8);
    w.front = o;    o = up256(o + fcap * M * 8);
    w.box_lo = o;   o = up256(o + (int64_t)box_cap * M * 4);
    w.box_hi = o;   o = up256(o + (int64_t)box_cap * M * 4);
    w.part_key = o; o = up256(o + kPartMax * 8);
    w.part_pos = o; o = up256(o + kPartMax * 4);
    w.rec = o;      o = up256(o + SCOOT_FANT_REC * 8);
    w.words = o;    o = up256(o + 16 * 4);
    w.fmap64 = o;   o = up256(o + 16 * 2 * 8);
    // the split copy of L^{-1} for the tensor-core posterior (when n_pad allows it)
    w.tcb_bytes = n_pad <= kMaxNpadTc ? scoot_tc_bsplit_bytes((int)n_pad, (int)M) : 0;
    w.tcb = o;      o = up256(o + w.tcb_bytes);
    w.bytes = o;
    return w;
}

int sm_count(int device) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, device);
    return v > 0 ? v : 1;
}

// An open session of sequential picks: the kernels' arguments and launch shapes.
struct Session {
    FantArgs a;
    int M;
    int64_t n;
    unsigned blocks;
    size_t pass_smem, pick_smem;
};

template <int M>
scoot_status set_attributes(scoot_ctx* ctx, Session& ss) {
    const FantArgs& a = ss.a;
    ss.pass_smem = (size_t)(2 * a.box_cap + a.n_mc) * 16 + (size_t)((a.q + 1) & ~1) * 8 + (size_t)M * a.n_pad * 4 +
                   (size_t)M * a.q * 4 + (size_t)M * 4 + (size_t)a.d * 4 + 16 +   // ... + culling:
                   (size_t)(a.n_mc / 8) * 16 + (size_t)a.n_mc * 4 + (size_t)kCullQueue * (2 * M * 4 + 8);
    ss.pick_smem = std::max((size_t)std::max(32 + a.slab_w, a.n_obs + 3 * a.q + 64 + a.q * a.q) * 8,
                            boxes_smem(a.front_cap, M, a.box_cap));
    int max_smem = 0;
    SCOOT_CUDA(ctx, cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, ctx->device));
    if (ss.pass_smem > (size_t)max_smem || ss.pick_smem > (size_t)max_smem)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "%d boxes and %d samples exceed the shared memory of a block",
                          a.box_cap, a.n_mc);
    SCOOT_CUDA(ctx, cudaFuncSetAttribute(fant_pass<M>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ss.pass_smem));
    SCOOT_CUDA(ctx, cudaFuncSetAttribute(fant_pick<M>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ss.pick_smem));
    SCOOT_CUDA(ctx, cudaFuncSetAttribute(fant_init<M>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ss.pick_smem));
    return SCOOT_OK;
}

Session* session_of(scoot_ctx* ctx) {
    return ctx->fant_session.size() == sizeof(Session) ? reinterpret_cast<Session*>(ctx->fant_session.data())
                                                        : nullptr;
}

}  // namespace

extern "C" {

scoot_status scoot_fantasy_work_bytes(const scoot_gp_layout* L, int64_t n, int32_t q, int32_t box_cap,
                                      int64_t* bytes) {
    if (!L || !bytes || n < 0 || box_cap < 1 || box_cap > kFantBoxMax) return SCOOT_EINVAL;
    if (q < 1 || q > SCOOT_MAX_Q) return SCOOT_EUNSUPPORTED;
    *bytes = work_layout(L, n, q, box_cap).bytes;
    return SCOOT_OK;
}

scoot_status scoot_fantasy_begin(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state, const void* fant_state,
                                 int32_t box_cap, const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                                 int64_t index_offset, const float* eps, int32_t n_mc, int32_t q, void* work,
                                 int64_t work_bytes, int64_t* idx, float* val, int32_t* count, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    ctx->fant_session.clear();
    if (!L || !state || !fant_state || !eps || !idx || !val || !count || !work)
        return scoot_fail(ctx, SCOOT_EINVAL, "a required pointer is NULL");
    if (!scoot_gp_layout_valid(L))
        return scoot_fail(ctx, SCOOT_EINVAL, "GP layout is not one made by scoot_gp_layout_init");
    const int M = L->n_obj;
    if (M < 2 || M > 4) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "fantasy picks need 2 <= M <= 4, got %d", M);
    if (q < 1 || q > SCOOT_MAX_Q) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "q = %d outside 1..%d", q, SCOOT_MAX_Q);
    if (n_mc < 1) return scoot_fail(ctx, SCOOT_EINVAL, "n_mc < 1");
    if (box_cap < 1 || box_cap > kFantBoxMax)
        return scoot_fail(ctx, SCOOT_EINVAL, "box_cap = %d outside 1..%d", box_cap, kFantBoxMax);
    if ((s = scoot_check_pool(ctx, cand, n, ld, L->d)) != SCOOT_OK) return s;
    if (n > 0x7FFFFFFFll) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "n >= 2^31");
    if (index_offset < 0 || index_offset + n > 0xFFFFFFFFll)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "global indices must lie below 2^32");
    const WorkLayout w = work_layout(L, n, q, box_cap);
    if (work_bytes < w.bytes)
        return scoot_fail(ctx, SCOOT_EINVAL, "work buffer of %lld bytes, %lld needed", (long long)work_bytes, (long long)w.bytes);
    if ((reinterpret_cast<uintptr_t>(work) & 255u) != 0) return scoot_fail(ctx, SCOOT_EINVAL, "work is not 256-byte aligned");
    if ((reinterpret_cast<uintptr_t>(fant_state) & 255u) != 0)
        return scoot_fail(ctx, SCOOT_EINVAL, "fant_state is not 256-byte aligned");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    char* wk = static_cast<char*>(work);
    Session ss;
    std::memset(&ss, 0, sizeof(ss));
    FantArgs& a = ss.a;
    a.n = n;
    a.ldc = n > 0 ? n : 1;
    a.index_offset = index_offset;
    if ((s = scoot_marks_begin(ctx, st)) != SCOOT_OK) return s;
    if (mask && n > 0) {
        ScootList lst;
        if ((s = scoot_compact(ctx, mask, n, nullptr, 0u, st, &lst)) != SCOOT_OK) return s;
        a.list = lst.list;
        a.n_list = lst.count;
        if ((s = scoot_mark(ctx, st, SCOOT_PHASE_COMPACT)) != SCOOT_OK) return s;
    }
    a.mean = reinterpret_cast<float*>(wk + w.mean);
    a.var = reinterpret_cast<float*>(wk + w.var);
    a.V = reinterpret_cast<float*>(wk + w.V);
    a.C = reinterpret_cast<float*>(wk + w.C);
    a.n_obs = L->n;
    a.n_pad = L->n_rb * 64;
    a.d = L->d;
    a.kernel = L->kernel;
    a.q = q;
    a.n_mc = n_mc;
    a.box_cap = box_cap;
    a.front_cap = L->n + q;
    a.gp = static_cast<const char*>(state);
    a.off_fmap = L->off_fmap;
    a.off_ils = L->off_ils;
    a.off_scal = L->off_scal;
    a.fant = static_cast<const char*>(fant_state);
    a.cand = cand;
    a.ld = ld;
    a.eps = eps;
    a.box_lo = reinterpret_cast<float*>(wk + w.box_lo);
    a.box_hi = reinterpret_cast<float*>(wk + w.box_hi);
    a.front = reinterpret_cast<double*>(wk + w.front);
    a.ctrl = reinterpret_cast<Ctrl*>(wk + w.ctrl);
    a.picked_pos = reinterpret_cast<int64_t*>(wk + w.picked);
    a.vp = reinterpret_cast<float*>(wk + w.vp);
    a.cxp = reinterpret_cast<float*>(wk + w.cxp);
    a.inv_s = reinterpret_cast<float*>(wk + w.inv_s);
    a.upick = reinterpret_cast<double*>(wk + w.upick);
    a.vpick = reinterpret_cast<double*>(wk + w.vpick);
    a.wf = reinterpret_cast<double*>(wk + w.wf);
    a.part = reinterpret_cast<double*>(wk + w.part);
    a.mupart = reinterpret_cast<double*>(wk + w.mupart);
    a.kpt = reinterpret_cast<double*>(wk + w.kpt);
    a.n_slab = pick_slabs(L->n);
    a.slab_w = (L->n + a.n_slab - 1) / a.n_slab;
    a.mupick = reinterpret_cast<double*>(wk + w.mupick);
    a.part_key = reinterpret_cast<uint64_t*>(wk + w.part_key);
    a.part_pos = reinterpret_cast<int32_t*>(wk + w.part_pos);
    a.rec = reinterpret_cast<uint64_t*>(wk + w.rec);
    a.pick_words = reinterpret_cast<uint32_t*>(wk + w.words);
    a.fmap64 = reinterpret_cast<double*>(wk + w.fmap64);
    a.out_idx = idx;
    a.out_val = val;
    a.out_count = count;
    a.err = ctx->d_err;
    if (n > 0) {
        s = scoot_posterior_whitened(ctx, L, state, cand, n, ld, a.list, a.n_list, reinterpret_cast<float*>(wk + w.mean),
                                     a.var, reinterpret_cast<float*>(wk + w.V), a.ldc,
                                     w.tcb_bytes > 0 ? static_cast<void*>(wk + w.tcb) : nullptr, st);
        if (s != SCOOT_OK) return s;
        if ((s = scoot_mark(ctx, st, SCOOT_PHASE_POSTERIOR)) != SCOOT_OK) return s;
    }
    ss.M = M;
    ss.n = n;
    // Enough blocks for many loads in flight per SM; the live count is read on the device.
    int64_t blocks = (n + kPassThreads - 1) / kPassThreads;
    const int64_t cap = std::min<int64_t>((int64_t)sm_count(ctx->device) * 8, kPartMax);
    ss.blocks = (unsigned)std::max<int64_t>(1, std::min(blocks, cap));
    switch (M) {
    case 2: s = set_attributes<2>(ctx, ss); break;
    case 3: s = set_attributes<3>(ctx, ss); break;
    default: s = set_attributes<4>(ctx, ss); break;
    }
    if (s != SCOOT_OK) return s;
    switch (M) {
    case 2: fant_init<2><<<1, kPickThreads, ss.pick_smem, st>>>(a); break;
    case 3: fant_init<3><<<1, kPickThreads, ss.pick_smem, st>>>(a); break;
    default: fant_init<4><<<1, kPickThreads, ss.pick_smem, st>>>(a); break;
    }
    SCOOT_LAUNCHED(ctx);
    if ((s = scoot_mark(ctx, st, SCOOT_PHASE_FANT_INIT)) != SCOOT_OK) return s;
    ctx->fant_session.resize(sizeof(Session));
    std::memcpy(ctx->fant_session.data(), &ss, sizeof(Session));
    return SCOOT_OK;
}

scoot_status scoot_fantasy_local_best(scoot_ctx* ctx, int32_t j, uint64_t* rec, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    Session* ss = session_of(ctx);
    if (!ss) return scoot_fail(ctx, SCOOT_EINVAL, "no open fantasy session (scoot_fantasy_begin)");
    if (j < 0 || j >= ss->a.q) return scoot_fail(ctx, SCOOT_EINVAL, "pick %d outside 0..%d", j, ss->a.q - 1);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    switch (ss->M) {
    case 2: fant_pass<2><<<ss->blocks, kPassThreads, ss->pass_smem, st>>>(ss->a, j); break;
    case 3: fant_pass<3><<<ss->blocks, kPassThreads, ss->pass_smem, st>>>(ss->a, j); break;
    default: fant_pass<4><<<ss->blocks, kPassThreads, ss->pass_smem, st>>>(ss->a, j); break;
    }
    SCOOT_LAUNCHED(ctx);
    if ((s = scoot_mark(ctx, st, SCOOT_PHASE_FANT_PASS)) != SCOOT_OK) return s;
    if (rec)
        SCOOT_CUDA(ctx, cudaMemcpyAsync(rec, ss->a.rec, SCOOT_FANT_REC * sizeof(uint64_t), cudaMemcpyDeviceToDevice, st));
    return SCOOT_OK;
}

scoot_status scoot_fantasy_commit(scoot_ctx* ctx, int32_t j, const uint64_t* recs, int32_t n_rec, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    Session* ss = session_of(ctx);
    if (!ss) return scoot_fail(ctx, SCOOT_EINVAL, "no open fantasy session (scoot_fantasy_begin)");
    if (j < 0 || j >= ss->a.q) return scoot_fail(ctx, SCOOT_EINVAL, "pick %d outside 0..%d", j, ss->a.q - 1);
    if (!recs || n_rec < 1) return scoot_fail(ctx, SCOOT_EINVAL, "no records");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const dim3 grid(ss->a.n_slab, ss->M);
    switch (ss->M) {
    case 2: fant_pick<2><<<grid, kPickThreads, ss->pick_smem, st>>>(ss->a, j, recs, n_rec); break;
    case 3: fant_pick<3><<<grid, kPickThreads, ss->pick_smem, st>>>(ss->a, j, recs, n_rec); break;
    default: fant_pick<4><<<grid, kPickThreads, ss->pick_smem, st>>>(ss->a, j, recs, n_rec); break;
    }
    SCOOT_LAUNCHED(ctx);
    return scoot_mark(ctx, st, SCOOT_PHASE_FANT_PICK);
}

scoot_status scoot_fantasy_end(scoot_ctx* ctx, float* var_out, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    Session* ss = session_of(ctx);
    if (!ss) return scoot_fail(ctx, SCOOT_EINVAL, "no open fantasy session (scoot_fantasy_begin)");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (var_out && ss->n > 0) {
        int64_t blocks = (ss->n + kPassThreads - 1) / kPassThreads;
        if (blocks > (int64_t)sm_count(ctx->device) * 8) blocks = (int64_t)sm_count(ctx->device) * 8;
        scatter_var<<<(unsigned)blocks, kPassThreads, 0, st>>>(ss->a.list, ss->a.n_list, ss->n, ss->a.ldc, ss->M,
                                                               ss->a.var, var_out, ss->n);
        SCOOT_LAUNCHED(ctx);
        if ((s = scoot_mark(ctx, st, SCOOT_PHASE_SCATTER)) != SCOOT_OK) return s;
    }
    ctx->fant_session.clear();
    return SCOOT_OK;
}

scoot_status scoot_suggest_fantasy(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state,
                                   const void* fant_state, int32_t box_cap, const uint32_t* cand, int64_t n,
                                   int64_t ld, const uint8_t* mask, const float* eps, int32_t n_mc, int32_t q,
                                   void* work, int64_t work_bytes, int64_t* idx, float* val, int32_t* count,
                                   float* var_out, void* stream) {
    scoot_status s = scoot_fantasy_begin(ctx, L, state, fant_state, box_cap, cand, n, ld, mask, 0, eps, n_mc, q, work,
                                         work_bytes, idx, val, count, stream);
    if (s != SCOOT_OK) return s;
    const uint64_t* rec = session_of(ctx)->a.rec;
    for (int j = 0; j < q; ++j) {
        if ((s = scoot_fantasy_local_best(ctx, j, nullptr, stream)) != SCOOT_OK) return s;
        if ((s = scoot_fantasy_commit(ctx, j, rec, 1, stream)) != SCOOT_OK) return s;
    }
    return scoot_fantasy_end(ctx, var_out, stream);
}

}  // extern "C"
