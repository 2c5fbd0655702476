// Device helpers shared by the scoring kernels (score.cu) and the fantasy
// kernels (fantasy.cu).
#pragma once

#include "internal.h"

namespace scoot_dev {

// The whitened rows V of the fantasy path, tiled by 32 list positions: the
// float4 group g (rows 4 g .. 4 g + 3) of objective m of list position p is
// float4 number ((p / 32) M + m) (n_pad / 4) 32 + 32 g + p mod 32.  The 32
// candidates of a warp then read or write 512 contiguous bytes per group,
// and each tile of 32 candidates is one contiguous block of HBM.
__host__ __device__ __forceinline__ int64_t vtile_index(int64_t p, int m, int g, int M, int n4) {
    return (((p >> 5) * M + m) * (int64_t)n4 + g) * 32 + (p & 31);
}

__device__ __forceinline__ float matern(float r, int kernel) {
    if (kernel == SCOOT_MATERN32) {
        const float a = 1.7320508075688772f * r;
        return (1.0f + a) * expf(-a);
    }
    const float a = 2.2360679774997896f * r;
    return fmaf(a, fmaf(a, 0.33333333333333333f, 1.0f), 1.0f) * expf(-a);
}

__device__ __forceinline__ float ei_value(float mu, float var, float ybest, float xi) {
    const float a = (mu - ybest) + xi;
    const float s = sqrtf(fmaxf(var, 0.0f));
    if (!(s > 0.0f)) return fmaxf(a, 0.0f);
    const float z = a / s;
    const float cdf = 0.5f * erfcf(-z * 0.70710678118654752f);
    const float pdf = 0.39894228040143268f * expf(-0.5f * z * z);
    return fmaf(a, cdf, s * pdf);
}

// Kumaraswamy CDF w(u) = 1 - (1 - u^a)^b (input warping), evaluated as
// -expm1(b log1p(-u^a)) so that small u^a keeps its relative accuracy.  Not
// inlined: the scoring kernels call it only for warped states, and inlining
// it raised the register pressure of their common, unwarped path.
static __device__ __noinline__ float kumaraswamy_cdf(float u, float a, float b) {
    u = fminf(fmaxf(u, 0.0f), 1.0f);
    const float ua = u > 0.0f ? exp2f(a * log2f(u)) : 0.0f;
    return -expm1f(b * log1pf(-ua));
}

// PI = P(f + xi > y+) = Phi((mu + xi - y+) / sigma); a step at sigma = 0.
__device__ __forceinline__ float pi_value(float mu, float var, float ybest, float xi) {
    const float a = (mu - ybest) + xi;
    const float s = sqrtf(fmaxf(var, 0.0f));
    if (!(s > 0.0f)) return a > 0.0f ? 1.0f : 0.0f;
    return 0.5f * erfcf(-(a / s) * 0.70710678118654752f);
}

// psi(a) = E[max(0, Y - a)] for Y ~ N(mu, sd^2), a finite:
// sd phi(z) + (mu - a) Phi(z) with z = (mu - a) / sd; max(0, mu - a) at sd = 0.
__device__ __forceinline__ float expected_excess(float mu, float sd, float a) {
    const float d = mu - a;
    if (!(sd > 0.0f)) return fmaxf(d, 0.0f);
    const float z = d / sd;
    const float cdf = 0.5f * erfcf(-z * 0.70710678118654752f);
    const float pdf = 0.39894228040143268f * expf(-0.5f * z * z);
    return fmaf(sd, pdf, d * cdf);
}

// Staging of the exact-EHVI boxes: the per-axis grids (axis j at
// grid_s[goff_j ..]) and the boxes' corner indices, validated against the
// grid sizes (an index beyond n_grid[j] is clamped and flagged).
__device__ __forceinline__ void stage_box_grid(const float* grid, int grid_cap, const int* n_grid, const uint32_t* corner,
                                               int n_boxes, int M, float* grid_s, uint32_t* corner_s, uint32_t* err) {
    int goff = 0;
    for (int j = 0; j < M; ++j) {
        for (int g = threadIdx.x; g < n_grid[j]; g += blockDim.x) grid_s[goff + g] = grid[j * grid_cap + g];
        goff += n_grid[j];
    }
    for (int e = threadIdx.x; e < n_boxes * M; e += blockDim.x) {
        const int j = e % M;
        uint32_t c = corner[e];
        const uint32_t lo = c & 0xFFFFu, hi = c >> 16, G = (uint32_t)n_grid[j];
        if (lo > G || hi > G) {
            atomicOr(err, 1u);  // SCOOT_DEVERR_INDEX
            c = (lo > G ? G : lo) | ((hi > G ? G : hi) << 16);
        }
        corner_s[e] = c;
    }
}

// UCB = mu + kappa * sigma.
__device__ __forceinline__ float ucb_value(float mu, float var, float kappa) {
    return fmaf(kappa, sqrtf(fmaxf(var, 0.0f)), mu);
}

// EHVI of one candidate: the mean over the S base samples of the hypervolume
// improvement, summed over boxes.  Boxes are float4 rows (lo, hi padded to
// four objectives), base samples float4 rows.  Samples are taken eight at a
// time so that each box is read from shared memory once per eight samples;
// padding samples sit at -inf and add nothing.
template <int M>
__device__ __forceinline__ float ehvi_value(const float* mu, const float* sd, const float4* blo,
                                            const float4* bhi, int n_boxes, const float4* eps,
                                            int n_mc) {
    constexpr int kCh = 8;
    float total = 0.0f;
    for (int s0 = 0; s0 < n_mc; s0 += kCh) {
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
    return total * (1.0f / (float)n_mc);
}

// Width that stands in for an unbounded side of a box on the first M-1
// objectives: a power of two, so scaling by it and by its inverse is exact;
// valid while every sample lies within 2^40 of the box's lower corner.
constexpr float kOpenWidth = 1099511627776.0f;  // 2^40

// Boxes open on the last objective in "saturated" form: for the first M-1
// objectives a_j = 1/w_j and b_j = -l_j/w_j (w_j the box width), and for the
// last one W = prod_j w_j and C = -l_last * W, so that a box's HVI term is
//   prod_{j<M-1} sat(y_j a_j + b_j) * max(y_last W + C, 0)
// (sat clamps to [0, 1]): one saturated FMA per bounded objective.
// Row b holds (a_0, b_0, a_1, b_1) and (W, W, C, C) as two float4 (M <= 3:
// the second row is two packed pairs for the f32x2 instructions).
__device__ __forceinline__ void stage_boxes_sat(const float* box_lo, const float* box_hi, int n_boxes, int M,
                                                float4* bs) {
    for (int b = threadIdx.x; b < n_boxes; b += blockDim.x) {
        float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        float W = 1.0f;
        for (int j = 0; j < M - 1; ++j) {
            const float l = box_lo[b * M + j], h = box_hi[b * M + j];
            const float w = h == INFINITY ? kOpenWidth : h - l;
            v[2 * j] = 1.0f / w;
            v[2 * j + 1] = -l / w;
            W *= w;
        }
        const float C = -box_lo[b * M + M - 1] * W;
        bs[2 * b] = make_float4(v[0], v[1], v[2], v[3]);
        bs[2 * b + 1] = make_float4(W, W, C, C);
    }
}

// Sum over samples first, first + stride, ... (chunks of eight) of the HVI of
// y_s = mu + sd * eps_s against boxes staged by stage_boxes_sat (M <= 3).
// Samples go in pairs through the packed f32x2 FMA and multiply (the same
// roundings as the scalar operations); the saturated FMAs and the maximum
// stay scalar.
template <int M>
__device__ __forceinline__ float ehvi_partial_sat(const float* mu, const float* sd, const float4* bs, int n_boxes,
                                                 const float4* eps, int n_mc, int first, int stride) {
    static_assert(M == 2 || M == 3, "the saturated form takes two or three objectives");
    constexpr int kCh = 8, kP = kCh / 2;
    float total = 0.0f;
    for (int s0 = first * kCh; s0 < n_mc; s0 += stride * kCh) {
        float ya[kCh], yb[kCh];  // the first M - 1 objectives (yb unused for M = 2)
        float2 yl[kP], acc[kP];  // the last objective and the sums, in pairs of samples
#pragma unroll
        for (int h = 0; h < kP; ++h) {
            float last[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int k = 2 * h + u;
                const bool in = s0 + k < n_mc;
                const float4 e = in ? eps[s0 + k] : make_float4(0.f, 0.f, 0.f, 0.f);
                ya[k] = in ? fmaf(sd[0], e.x, mu[0]) : -INFINITY;
                yb[k] = M > 2 ? (in ? fmaf(sd[1], e.y, mu[1]) : -INFINITY) : 0.0f;
                last[u] = in ? fmaf(sd[M - 1], M > 2 ? e.z : e.y, mu[M - 1]) : -INFINITY;
            }
            yl[h] = make_float2(last[0], last[1]);
            acc[h] = make_float2(0.0f, 0.0f);
        }
        for (int b = 0; b < n_boxes; ++b) {
            const float4 q0 = bs[2 * b], q1 = bs[2 * b + 1];
            const float2 Wp = make_float2(q1.x, q1.y), Cp = make_float2(q1.z, q1.w);
#pragma unroll
            for (int h = 0; h < kP; ++h) {
                float2 p = make_float2(__saturatef(fmaf(ya[2 * h], q0.x, q0.y)),
                                       __saturatef(fmaf(ya[2 * h + 1], q0.x, q0.y)));
                if (M > 2)
                    p = __fmul2_rn(p, make_float2(__saturatef(fmaf(yb[2 * h], q0.z, q0.w)),
                                                  __saturatef(fmaf(yb[2 * h + 1], q0.z, q0.w))));
                const float2 t = __ffma2_rn(yl[h], Wp, Cp);
                acc[h] = __ffma2_rn(p, make_float2(fmaxf(t.x, 0.0f), fmaxf(t.y, 0.0f)), acc[h]);
            }
        }
#pragma unroll
        for (int h = 0; h < kP; ++h) total += acc[h].x + acc[h].y;
    }
    return total;
}

// True (in every thread) when the saturated form is exact for the staged
// boxes: every box is open on the last objective, M <= 3, and every lower
// corner lies within 2^30 of zero.  The form folds one open width 2^40 per
// open leading axis into W, so W <= 2^80 and |C| <= 2^110 for M <= 3 (finite
// in fp32 for samples within 2^40 of the corner); with M = 4 the last box
// would carry W = 2^120, whose products with y_last and l_last overflow (and
// whose reciprocal factors underflow) at ordinary objective scales, so M = 4
// always takes the general form.
__device__ __forceinline__ bool boxes_fast(const float4* blo, const float4* bhi, int n_boxes, int M) {
    int ok = M <= 3;
    constexpr float kCornerMax = 1073741824.0f;  // 2^30
    for (int b = threadIdx.x; b < n_boxes && ok; b += blockDim.x) {
        const float4 h = bhi[b], l = blo[b];
        ok &= (M == 2 ? h.y : (M == 3 ? h.z : h.w)) == INFINITY;
        ok &= fabsf(l.x) < kCornerMax && fabsf(l.y) < kCornerMax && (M < 3 || fabsf(l.z) < kCornerMax);
    }
    return __syncthreads_and(ok) != 0;
}

// Boxes ([B][M] lower and upper bounds) and base samples ([S][M]) into shared
// memory as float4 rows padded to four objectives.
__device__ __forceinline__ void stage_boxes(const float* box_lo, const float* box_hi, int n_boxes, const float* eps_in,
                                            int n_mc, int M, float4* blo, float4* bhi, float4* eps) {
    for (int b = threadIdx.x; b < n_boxes; b += blockDim.x) {
        float l[4] = {0.f, 0.f, 0.f, 0.f}, h[4] = {0.f, 0.f, 0.f, 0.f};
        for (int j = 0; j < M; ++j) {
            l[j] = box_lo[b * M + j];
            h[j] = box_hi[b * M + j];
        }
        blo[b] = make_float4(l[0], l[1], l[2], l[3]);
        bhi[b] = make_float4(h[0], h[1], h[2], h[3]);
    }
    for (int s = threadIdx.x; s < n_mc; s += blockDim.x) {
        float e[4] = {0.f, 0.f, 0.f, 0.f};
        for (int j = 0; j < M; ++j) e[j] = eps_in[s * M + j];
        eps[s] = make_float4(e[0], e[1], e[2], e[3]);
    }
}

// Covariance-input coordinate of one stored parameter value (Section 4.3 with
// the feature map of include/scoot.h): log scale for integer log-uniform
// parameters, linear for integer uniform and continuous ones, the category
// index for categoricals; a and b are the offset and scale of the map.
__device__ __forceinline__ float feature_of(uint32_t w, int kind, float a, float b) {
    if (kind == SCOOT_INT_LOG) return (logf((float)(int32_t)w) - a) * b;
    if (kind == SCOOT_INT_UNIFORM) return ((float)(int32_t)w - a) * b;
    if (kind == SCOOT_CONTINUOUS) return (__uint_as_float(w) - a) * b;
    return (float)(int32_t)w;
}


// Selection key of a candidate (Section 4.7 order): the high word is the
// value mapped to an order-preserving unsigned integer, the low word is
// 0xFFFFFFFF - index, so a larger key is a larger value or, on equal
// values, a lower index.  -0 and +0 are one value (the comparison of the
// selection rule is numeric), so -0 is mapped to +0 first.  0 is never a key
// of an eligible candidate.
__device__ __forceinline__ uint64_t make_key(float v, uint32_t idx) {
    uint32_t b = __float_as_uint(v);
    if (b == 0x80000000u) b = 0u;
    b = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
    return ((uint64_t)b << 32) | (uint64_t)(0xFFFFFFFFu - idx);
}

__device__ __forceinline__ float key_value(uint64_t k) {
    uint32_t b = (uint32_t)(k >> 32);
    b = (b & 0x80000000u) ? (b & 0x7FFFFFFFu) : ~b;
    return __uint_as_float(b);
}

__device__ __forceinline__ int64_t key_index(uint64_t k) {
    return (int64_t)(0xFFFFFFFFu - (uint32_t)(k & 0xFFFFFFFFu));
}

}  // namespace scoot_dev
