// Quasi-random configurations for the tuning loop around the scoring path
// (Algorithm 1's initial design and Section 4.6's shortfall fill, both drawn
// from a Sobol sequence), the selection of the first feasible ones, and
// Algorithm 1's feasibility-threshold controller.
//
// Sobol directions: dimension 0 is the van der Corput sequence; dimension
// j >= 1 takes the j-th primitive polynomial over GF(2) (by degree, then by
// its middle coefficients read as a binary number, a_1 most significant)
// with unit initial direction integers m_1 = ... = m_s = 1 and the
// recurrence m_k = 2 a_1 m_(k-1) ^ 4 a_2 m_(k-2) ^ ... ^ 2^(s-1) a_(s-1)
// m_(k-s+1) ^ 2^s m_(k-s) ^ m_(k-s); V_k = m_k 2^(32-k).  Point i is the
// xor of V_k over the set bits k - 1 of i.
#include <cmath>
#include <cstring>
#include <vector>

#include "internal.h"

namespace {

constexpr int kSobolThreads = 256;
constexpr int kFirstThreads = 1024;

struct SobolArgs {
    uint32_t V[SCOOT_MAX_DIM][32];  // V[j][k - 1]
    int32_t kind[SCOOT_MAX_DIM];
    int32_t n_choices[SCOOT_MAX_DIM];
    double lo[SCOOT_MAX_DIM], hi[SCOOT_MAX_DIM];
    double log_lo[SCOOT_MAX_DIM], log_span[SCOOT_MAX_DIM];
    int32_t d;
    int64_t skip, n, ld;
    uint32_t* cand;
};

// x^k mod poly (degree s) over GF(2), as a bit mask.
uint32_t mulx_mod(uint32_t p, uint32_t poly, int s) {
    p <<= 1;
    if ((p >> s) & 1u) p ^= poly;
    return p;
}

// x has multiplicative order 2^s - 1 modulo poly.
bool primitive(uint32_t poly, int s) {
    const uint32_t e = (1u << s) - 1u;
    uint32_t x = 1;
    for (uint32_t k = 1; k <= e; ++k) {
        x = mulx_mod(x, poly, s);
        if (x == 1u) return k == e;
    }
    return false;
}

// Direction integers of the first d dimensions.
void sobol_directions(int d, uint32_t (*V)[32]) {
    for (int k = 1; k <= 32; ++k) V[0][k - 1] = 1u << (32 - k);
    int j = 1;
    for (int s = 1; j < d; ++s) {
        for (uint32_t a = 0; a < (1u << (s - 1)) && j < d; ++a) {
            const uint32_t poly = (1u << s) | (a << 1) | 1u;
            if (!primitive(poly, s)) continue;
            uint64_t m[33] = {0};
            for (int k = 1; k <= 32; ++k) {
                if (k <= s) {
                    m[k] = 1;
                } else {
                    uint64_t v = m[k - s] ^ (m[k - s] << s);
                    for (int i = 1; i < s; ++i)
                        if ((a >> (s - 1 - i)) & 1u) v ^= m[k - i] << i;
                    m[k] = v;
                }
                V[j][k - 1] = (uint32_t)(m[k] << (32 - k));
            }
            ++j;
        }
    }
}

// One thread per point: the Sobol integers of its dimensions, mapped in
// fp64 onto each parameter's range and stored as the pool's words.
__global__ void __launch_bounds__(kSobolThreads) sobol_kernel(const __grid_constant__ SobolArgs a) {
    for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < a.n; r += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t i = (uint32_t)(a.skip + r);
        for (int j = 0; j < a.d; ++j) {
            uint32_t x = 0;
            for (uint32_t b = i, k = 0; b; b >>= 1, ++k)
                if (b & 1u) x ^= a.V[j][k];
            const double u = (double)x * 2.3283064365386963e-10;  // 2^-32
            uint32_t w;
            // Explicit roundings (no fused multiply-add), in the order the
            // mapping is defined, so that the words do not depend on contraction.
            switch (a.kind[j]) {
            case SCOOT_INT_LOG: {
                double v = rint(exp(__dadd_rn(a.log_lo[j], __dmul_rn(u, a.log_span[j]))));
                v = fmin(fmax(v, a.lo[j]), a.hi[j]);
                w = (uint32_t)(int32_t)v;
                break;
            }
            case SCOOT_INT_UNIFORM: {
                const double range = __dadd_rn(__dsub_rn(a.hi[j], a.lo[j]), 1.0);
                const double v = fmin(__dadd_rn(a.lo[j], floor(__dmul_rn(u, range))), a.hi[j]);
                w = (uint32_t)(int32_t)v;
                break;
            }
            case SCOOT_CATEGORICAL:
                w = (uint32_t)(int32_t)floor(__dmul_rn(u, (double)a.n_choices[j]));
                break;
            default:
                w = __float_as_uint(__double2float_rn(__dadd_rn(a.lo[j], __dmul_rn(u, __dsub_rn(a.hi[j], a.lo[j])))));
                break;
            }
            a.cand[(int64_t)j * a.ld + r] = w;
        }
    }
}

// One block: the first `need` positions p < n with mask[p] != 0, in
// increasing order, into idx; *count receives how many there were (<= need).
// The block walks the mask in rounds of kFirstThreads positions with a
// block-wide exclusive scan of the set flags.
__global__ void __launch_bounds__(kFirstThreads)
first_set_kernel(const uint8_t* __restrict__ mask, int64_t n, int32_t need, int64_t* __restrict__ idx,
                 int32_t* __restrict__ count) {
    __shared__ int warp_sum[kFirstThreads / 32];
    __shared__ int base;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) base = 0;
    __syncthreads();
    for (int64_t p0 = 0; p0 < n; p0 += kFirstThreads) {
        const int64_t p = p0 + tid;
        const bool set = p < n && mask[p] != 0;
        const unsigned int b = __ballot_sync(0xffffffffu, set);
        if (lane == 0) warp_sum[warp] = __popc(b);
        __syncthreads();
        int before = 0, total = 0;
        for (int w = 0; w < kFirstThreads / 32; ++w) {
            before += w < warp ? warp_sum[w] : 0;
            total += warp_sum[w];
        }
        const int rank = base + before + __popc(b & ((1u << lane) - 1u));
        if (set && rank < need) idx[rank] = p;
        __syncthreads();  // every thread has read base and warp_sum
        if (tid == 0) base += total;
        __syncthreads();
        if (base >= need) break;  // the same in every thread
    }
    if (tid == 0) *count = base < need ? base : need;
    for (int r = base + tid; r < need; r += kFirstThreads) idx[r] = -1;
}

int sm_count(int device) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, device);
    return v > 0 ? v : 1;
}

}  // namespace

extern "C" {

scoot_status scoot_sobol_configs(scoot_ctx* ctx, const scoot_param* h_space, int32_t d, int64_t skip, int64_t n,
                                 uint32_t* cand, int64_t ld, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (!h_space) return scoot_fail(ctx, SCOOT_EINVAL, "h_space is NULL");
    if (d < 1 || d > SCOOT_MAX_DIM) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "d = %d outside 1..%d", d, SCOOT_MAX_DIM);
    if (skip < 0 || n < 0) return scoot_fail(ctx, SCOOT_EINVAL, "skip and n must be >= 0");
    if (skip + n > 0xFFFFFFFFll) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "points beyond index 2^32 - 1");
    if (n == 0) return SCOOT_OK;
    if (!cand || ld < n) return scoot_fail(ctx, SCOOT_EINVAL, "cand is NULL or ld = %lld < n", (long long)ld);
    SobolArgs a;
    std::memset(&a, 0, sizeof(a));
    sobol_directions(d, a.V);
    for (int c = 0; c < d; ++c) {
        const scoot_param& p = h_space[c];
        a.kind[c] = p.kind;
        a.n_choices[c] = p.n_choices;
        a.lo[c] = p.lo;
        a.hi[c] = p.hi;
        if (p.kind == SCOOT_INT_LOG) {
            if (!(p.lo > 0.0f) || !(p.hi >= p.lo)) return scoot_fail(ctx, SCOOT_EINVAL, "parameter %d: bad log range", c);
            a.log_lo[c] = std::log((double)p.lo);
            a.log_span[c] = std::log((double)p.hi) - std::log((double)p.lo);
        } else if (p.kind == SCOOT_CATEGORICAL) {
            if (p.n_choices < 1) return scoot_fail(ctx, SCOOT_EINVAL, "parameter %d: n_choices < 1", c);
        } else if (p.kind != SCOOT_INT_UNIFORM && p.kind != SCOOT_CONTINUOUS) {
            return scoot_fail(ctx, SCOOT_EINVAL, "parameter %d: kind %d", c, p.kind);
        } else if (!(p.hi >= p.lo)) {
            return scoot_fail(ctx, SCOOT_EINVAL, "parameter %d: hi < lo", c);
        }
    }
    a.d = d;
    a.skip = skip;
    a.n = n;
    a.ld = ld;
    a.cand = cand;
    int64_t blocks = (n + kSobolThreads - 1) / kSobolThreads;
    const int64_t cap = (int64_t)sm_count(ctx->device) * 8;
    if (blocks > cap) blocks = cap;
    sobol_kernel<<<(unsigned)blocks, kSobolThreads, 0, static_cast<cudaStream_t>(stream)>>>(a);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

scoot_status scoot_first_feasible(scoot_ctx* ctx, const uint8_t* mask, int64_t n, int32_t need, int64_t* idx,
                                  int32_t* count, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (n < 0 || n > 0x7FFFFFFFll) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "n = %lld outside 0..2^31 - 1", (long long)n);
    if (need < 1 || need > SCOOT_MAX_Q) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "need = %d outside 1..%d", need, SCOOT_MAX_Q);
    if (!idx || !count || (n > 0 && !mask)) return scoot_fail(ctx, SCOOT_EINVAL, "mask, idx or count is NULL");
    first_set_kernel<<<1, kFirstThreads, 0, static_cast<cudaStream_t>(stream)>>>(mask, n, need, idx, count);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

scoot_status scoot_ucb_beta(int32_t t, double* beta) {
    if (!beta || t < 1) return SCOOT_EINVAL;
    const double tt = (double)t * (double)t;
    const double delta = 1.0 / tt;
    *beta = 2.0 * std::log(tt * M_PI * M_PI / (6.0 * delta));
    return SCOOT_OK;
}

scoot_status scoot_standardize(const float* h_y, int32_t n_obj, int32_t n, float* h_y_std, float* h_ref,
                               float ref_margin) {
    if (!h_y || !h_y_std || n_obj < 1 || n < 1) return SCOOT_EINVAL;
    for (int m = 0; m < n_obj; ++m) {
        const float* y = h_y + (size_t)m * n;
        double mean = 0.0;
        for (int i = 0; i < n; ++i) {
            if (!std::isfinite(y[i])) return SCOOT_EINVAL;
            mean += y[i];
        }
        mean /= n;
        double var = 0.0;
        for (int i = 0; i < n; ++i) var += ((double)y[i] - mean) * ((double)y[i] - mean);
        const double sd = std::fmax(std::sqrt(var / n), 1e-12);
        float lo = INFINITY;
        for (int i = 0; i < n; ++i) {
            h_y_std[(size_t)m * n + i] = (float)(((double)y[i] - mean) / sd);
            lo = std::fmin(lo, h_y_std[(size_t)m * n + i]);
        }
        if (h_ref) h_ref[m] = lo - ref_margin;
    }
    return SCOOT_OK;
}

scoot_status scoot_delta_update(double* delta, int32_t* count, int32_t k, int32_t any_invalid) {
    if (!delta || !count || k < 0) return SCOOT_EINVAL;
    constexpr double kStep = 0.05;
    if (any_invalid) {
        *delta = std::fmin(0.75, std::fmax(0.5, *delta + kStep));
        *count = 0;
    } else {
        *count += k;
        if (*count >= 5) {
            *delta = std::fmax(0.25, *delta - kStep);
            *count -= 5;
        }
    }
    return SCOOT_OK;
}

}  // extern "C"
