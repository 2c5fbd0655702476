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
// Device: one posterior pass storing mean, variance and V for the live
// candidates (list-position order); per pick an EHVI pass, an argmax and a
// downdate pass that reads V once.  Host, fp64, per pick: the picked point's
// features, k(X, x_p), v_p, mu(x_p), the c_l(x_p) and s_j.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <vector>

#include "device_common.cuh"
#include "internal.h"

namespace {

using namespace scoot_dev;

constexpr int kFThreads = 128;
constexpr int kBoxCap = 4096;
constexpr int kArgBlocks = 1024;

struct FantArgs {
    const int32_t* list;          // list position -> candidate index (NULL: identity)
    int64_t n_live, ldc;
    const float* mean;            // [M][ldc]
    float* var;                   // [M][ldc]
    const float* V;               // [M][n_pad][ldc]
    float* C;                     // [q][M][ldc]
    const float* vp;              // [M][n_pad]
    const float* cxp;             // [M][q]
    const float* inv_s;           // [M]
    const int64_t* picked;
    int32_t n_picked, n_pad, q, j;
    float* acq;                   // [ldc]
    const char* state;
    int64_t off_fmap, off_ils, off_scal;
    int32_t n_obs, d, kernel;
    const uint32_t* cand;
    int64_t ld, p;
    const float* box_lo;
    const float* box_hi;
    int32_t n_boxes;
    const float* eps;
    int32_t n_mc;
    uint64_t* partial;
    uint64_t* best;
};

template <int M>
__global__ void __launch_bounds__(kFThreads) fant_ehvi(const __grid_constant__ FantArgs a) {
    extern __shared__ __align__(16) float sm[];
    float4* blo = reinterpret_cast<float4*>(sm);
    float4* bhi = blo + a.n_boxes;
    float4* epsv = bhi + a.n_boxes;
    stage_boxes(a.box_lo, a.box_hi, a.n_boxes, a.eps, a.n_mc, M, blo, bhi, epsv);
    __syncthreads();
    for (int64_t pos = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; pos < a.n_live;
         pos += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = a.list ? (int64_t)a.list[pos] : pos;
        bool taken = false;
        for (int k = 0; k < a.n_picked; ++k) taken |= a.picked[k] == i;
        float v = -INFINITY;
        if (!taken) {
            float mu[M], sd[M];
#pragma unroll
            for (int m = 0; m < M; ++m) {
                mu[m] = a.mean[(int64_t)m * a.ldc + pos];
                sd[m] = sqrtf(fmaxf(a.var[(int64_t)m * a.ldc + pos], 0.0f));
            }
            v = ehvi_value<M>(mu, sd, blo, bhi, a.n_boxes, epsv, a.n_mc);
        }
        a.acq[pos] = v;
    }
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
    for (int o = 16; o > 0; o >>= 1) {
        const uint64_t w = __shfl_xor_sync(0xffffffffu, v, o);
        v = w > v ? w : v;
    }
    return v;
}

__device__ __forceinline__ uint64_t block_max_u64(uint64_t v) {
    __shared__ uint64_t wm[32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_max_u64(v);
    if (lane == 0) wm[warp] = v;
    __syncthreads();
    v = threadIdx.x < (blockDim.x >> 5) ? wm[threadIdx.x] : 0ull;
    if (warp == 0) v = warp_max_u64(v);
    return v;  // valid in thread 0
}

// Argmax over list positions with the selection key of the candidate index.
__global__ void __launch_bounds__(kFThreads) fant_argmax1(const __grid_constant__ FantArgs a) {
    uint64_t best = 0ull;
    for (int64_t pos = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; pos < a.n_live;
         pos += (int64_t)gridDim.x * blockDim.x) {
        const float v = a.acq[pos];
        if (!(v != v) && v != -INFINITY) {
            const uint64_t k = make_key(v, (uint32_t)(a.list ? a.list[pos] : pos));
            best = k > best ? k : best;
        }
    }
    best = block_max_u64(best);
    if (threadIdx.x == 0) a.partial[blockIdx.x] = best;
}

__global__ void __launch_bounds__(kFThreads) fant_argmax2(const __grid_constant__ FantArgs a, int n_partial) {
    uint64_t best = 0ull;
    for (int k = threadIdx.x; k < n_partial; k += blockDim.x) best = a.partial[k] > best ? a.partial[k] : best;
    best = block_max_u64(best);
    if (threadIdx.x == 0) *a.best = best;
}

// Variance downdate of every live candidate for pick j (see the file comment).
template <int M>
__global__ void __launch_bounds__(kFThreads) fant_update(const __grid_constant__ FantArgs a) {
    const float* fmap = reinterpret_cast<const float*>(a.state + a.off_fmap);
    const float* gils = reinterpret_cast<const float*>(a.state + a.off_ils);
    const float* gscal = reinterpret_cast<const float*>(a.state + a.off_scal);
    for (int64_t pos = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; pos < a.n_live;
         pos += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = a.list ? (int64_t)a.list[pos] : pos;
        float r2[M];
#pragma unroll
        for (int m = 0; m < M; ++m) r2[m] = 0.0f;
        for (int c = 0; c < a.d; ++c) {
            const int kind = (int)fmap[c * 4];
            const int64_t col = (int64_t)fmap[c * 4 + 3];  // features are in feature order
            const float ux = feature_of(__ldg(a.cand + col * a.ld + i), kind, fmap[c * 4 + 1], fmap[c * 4 + 2]);
            const float up = feature_of(__ldg(a.cand + col * a.ld + a.p), kind, fmap[c * 4 + 1], fmap[c * 4 + 2]);
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
            const float* vrow = a.V + (int64_t)m * a.n_pad * a.ldc + pos;
            const float* vp = a.vp + m * a.n_pad;
            float dot = 0.0f;
            for (int row = 0; row < a.n_obs; ++row) dot = fmaf(vrow[(int64_t)row * a.ldc], vp[row], dot);
            float cc = 0.0f;
            for (int l = 0; l < a.j; ++l) cc = fmaf(a.C[((int64_t)l * M + m) * a.ldc + pos], a.cxp[m * a.q + l], cc);
            const float c = (k - dot - cc) * a.inv_s[m];
            a.C[((int64_t)a.j * M + m) * a.ldc + pos] = c;
            float* vv = a.var + (int64_t)m * a.ldc + pos;
            *vv = fmaxf(*vv - c * c, 0.0f);
        }
    }
}

__global__ void __launch_bounds__(kFThreads)
scatter_var(const int32_t* list, int64_t n_live, int64_t ldc, int M, const float* var, float* out, int64_t ldo) {
    for (int64_t pos = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; pos < n_live;
         pos += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = list ? (int64_t)list[pos] : pos;
        for (int m = 0; m < M; ++m) out[(int64_t)m * ldo + i] = var[(int64_t)m * ldc + pos];
    }
}

struct WorkLayout {
    int64_t mean, var, V, C, acq, picked, vp, cxp, inv_s, box_lo, box_hi, partial, best, bytes;
};

int64_t up256(int64_t x) { return (x + 255) / 256 * 256; }

WorkLayout work_layout(const scoot_gp_layout* L, int64_t n, int q) {
    const int64_t M = L->n_obj, n_pad = (int64_t)L->n_rb * 64;
    WorkLayout w;
    int64_t o = 0;
    w.mean = o;    o = up256(o + M * n * 4);
    w.var = o;     o = up256(o + M * n * 4);
    w.V = o;       o = up256(o + M * n_pad * n * 4);
    w.C = o;       o = up256(o + (int64_t)q * M * n * 4);
    w.acq = o;     o = up256(o + n * 4);
    w.picked = o;  o = up256(o + (int64_t)q * 8);
    w.vp = o;      o = up256(o + M * n_pad * 4);
    w.cxp = o;     o = up256(o + M * q * 4);
    w.inv_s = o;   o = up256(o + M * 4);
    w.box_lo = o;  o = up256(o + (int64_t)kBoxCap * M * 4);
    w.box_hi = o;  o = up256(o + (int64_t)kBoxCap * M * 4);
    w.partial = o; o = up256(o + kArgBlocks * 8);
    w.best = o;    o = up256(o + 8);
    w.bytes = o;
    return w;
}

int sm_count(int device) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, device);
    return v > 0 ? v : 1;
}

struct Pick {
    std::vector<double> u;                  // features
    std::vector<std::vector<double>> v;     // [M][n] whitened covariance row
    std::vector<std::vector<double>> c;     // [M][l < j] c_l(x_p)
    std::vector<double> s;                  // [M] s_j
};

template <int M>
scoot_status run_picks(scoot_ctx* ctx, const scoot_gp_layout* L, FantArgs a, const std::vector<HostGP>& gps,
                       const scoot_param* h_space, const uint32_t* cand, int64_t ld, const float* h_y,
                       const float* h_ref, int32_t q, char* work, const WorkLayout& w, int64_t* h_idx,
                       float* h_val, int32_t* h_count, cudaStream_t st) {
    const int n = L->n, d = L->d, n_pad = L->n_rb * 64;
    std::vector<float> Y((size_t)M * n);
    std::memcpy(Y.data(), h_y, Y.size() * sizeof(float));
    int n_pts = n;
    std::vector<float> lo((size_t)kBoxCap * M), hi((size_t)kBoxCap * M);
    std::vector<float> vp_h((size_t)M * n_pad), cxp_h((size_t)M * q), inv_s_h(M);
    std::vector<Pick> picks;
    std::vector<uint32_t> words(d);
    const int sms = sm_count(ctx->device);
    int64_t blocks = (a.n_live + kFThreads - 1) / kFThreads;
    if (blocks > (int64_t)sms * 16) blocks = (int64_t)sms * 16;
    if (blocks < 1) blocks = 1;
    int arg_blocks = (int)std::min<int64_t>(blocks, kArgBlocks);
    *h_count = 0;
    for (int j = 0; j < q; ++j) {
        // Boxes of the front with the fantasised points added.
        int32_t nb = 0, fs = 0;
        scoot_status s = scoot_boxes_build(Y.data(), n_pts, M, h_ref, kBoxCap, lo.data(), hi.data(), &nb, &fs);
        if (s != SCOOT_OK) return scoot_fail(ctx, s, "box decomposition of the fantasised front failed (%d boxes)", nb);
        if ((size_t)(2 * nb + a.n_mc) * 16 > 160 * 1024)
            return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "%d boxes and %d samples exceed the shared-memory budget", nb, a.n_mc);
        SCOOT_CUDA(ctx, cudaMemcpyAsync(work + w.box_lo, lo.data(), (size_t)nb * M * 4, cudaMemcpyHostToDevice, st));
        SCOOT_CUDA(ctx, cudaMemcpyAsync(work + w.box_hi, hi.data(), (size_t)nb * M * 4, cudaMemcpyHostToDevice, st));
        a.n_boxes = nb;
        a.n_picked = j;
        a.j = j;
        const size_t smem = (size_t)(2 * nb + a.n_mc) * 16;
        SCOOT_CUDA(ctx, cudaFuncSetAttribute(fant_ehvi<M>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        fant_ehvi<M><<<(unsigned)blocks, kFThreads, smem, st>>>(a);
        SCOOT_LAUNCHED(ctx);
        fant_argmax1<<<arg_blocks, kFThreads, 0, st>>>(a);
        SCOOT_LAUNCHED(ctx);
        fant_argmax2<<<1, kFThreads, 0, st>>>(a, arg_blocks);
        SCOOT_LAUNCHED(ctx);
        uint64_t key = 0;
        SCOOT_CUDA(ctx, cudaMemcpyAsync(&key, work + w.best, 8, cudaMemcpyDeviceToHost, st));
        SCOOT_CUDA(ctx, cudaStreamSynchronize(st));
        if (key == 0) break;
        const int64_t p = (int64_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFu));
        uint32_t vb = (uint32_t)(key >> 32);
        vb = (vb & 0x80000000u) ? (vb & 0x7FFFFFFFu) : ~vb;
        float val;
        std::memcpy(&val, &vb, 4);
        h_idx[j] = p;
        h_val[j] = val;
        *h_count = j + 1;
        if (j + 1 == q) break;  // no later pick needs this one's fantasy
        // The picked configuration, on the host.
        SCOOT_CUDA(ctx, cudaMemcpy2DAsync(words.data(), 4, cand + p, (size_t)ld * 4, 4, d, cudaMemcpyDeviceToHost, st));
        SCOOT_CUDA(ctx, cudaStreamSynchronize(st));
        Pick pk;
        pk.u.resize(d);
        if (!scoot_host_features(h_space, d, words.data(), 1, 0, pk.u.data()))
            return scoot_fail(ctx, SCOOT_EINVAL, "picked configuration %lld has an invalid value", (long long)p);
        pk.v.assign(M, std::vector<double>(n));
        pk.c.assign(M, std::vector<double>(j));
        pk.s.assign(M, 0.0);
        std::vector<double> kx(n), mus(M);
        for (int m = 0; m < M; ++m) {
            const HostGP& g = gps[m];
            g.kstar(pk.u.data(), kx.data());
            g.solve_lower(kx.data(), pk.v[m].data());
            double mu = 0.0, vv = 0.0;
            for (int t = 0; t < n; ++t) {
                mu += kx[t] * g.alpha[t];
                vv += pk.v[m][t] * pk.v[m][t];
            }
            mus[m] = mu;  // kriging believer: the fantasised value is the posterior mean
            double var = g.sf2 - vv;
            for (int l = 0; l < j; ++l) {
                const Pick& pl = picks[l];
                double num = g.cov(pk.u.data(), pl.u.data());
                for (int t = 0; t < n; ++t) num -= pk.v[m][t] * pl.v[m][t];
                for (int t = 0; t < l; ++t) num -= pk.c[m][t] * pl.c[m][t];
                pk.c[m][l] = pl.s[m] > 0.0 ? num / pl.s[m] : 0.0;
                var -= pk.c[m][l] * pk.c[m][l];
            }
            pk.s[m] = std::sqrt(std::max(var, 0.0) + g.tau2);
            for (int t = 0; t < n_pad; ++t) vp_h[(size_t)m * n_pad + t] = t < n ? (float)pk.v[m][t] : 0.0f;
            for (int l = 0; l < q; ++l) cxp_h[(size_t)m * q + l] = l < j ? (float)pk.c[m][l] : 0.0f;
            inv_s_h[m] = pk.s[m] > 0.0 ? (float)(1.0 / pk.s[m]) : 0.0f;
        }
        // The fantasised observation joins the front.
        std::vector<float> Yn((size_t)M * (n_pts + 1));
        for (int m = 0; m < M; ++m) {
            std::memcpy(&Yn[(size_t)m * (n_pts + 1)], &Y[(size_t)m * n_pts], (size_t)n_pts * sizeof(float));
            Yn[(size_t)m * (n_pts + 1) + n_pts] = (float)mus[m];
        }
        Y.swap(Yn);
        n_pts += 1;
        picks.push_back(pk);
        SCOOT_CUDA(ctx, cudaMemcpyAsync(work + w.vp, vp_h.data(), vp_h.size() * 4, cudaMemcpyHostToDevice, st));
        SCOOT_CUDA(ctx, cudaMemcpyAsync(work + w.cxp, cxp_h.data(), cxp_h.size() * 4, cudaMemcpyHostToDevice, st));
        SCOOT_CUDA(ctx, cudaMemcpyAsync(work + w.inv_s, inv_s_h.data(), inv_s_h.size() * 4, cudaMemcpyHostToDevice, st));
        SCOOT_CUDA(ctx, cudaMemcpyAsync(work + w.picked + 8 * (size_t)j, &h_idx[j], 8, cudaMemcpyHostToDevice, st));
        a.p = p;
        fant_update<M><<<(unsigned)blocks, kFThreads, 0, st>>>(a);
        SCOOT_LAUNCHED(ctx);
    }
    return SCOOT_OK;
}

}  // namespace

extern "C" {

scoot_status scoot_fantasy_work_bytes(const scoot_gp_layout* L, int64_t n, int32_t q, int64_t* bytes) {
    if (!L || !bytes || n < 0 || q < 1 || q > SCOOT_MAX_Q) return SCOOT_EINVAL;
    *bytes = work_layout(L, n, q).bytes;
    return SCOOT_OK;
}

scoot_status scoot_suggest_fantasy(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state,
                                   const scoot_param* h_space, const uint32_t* h_x_obs, int64_t ld_obs,
                                   const float* h_y, const float* h_lengthscale, const float* h_signal_var,
                                   const float* h_noise_var, const uint32_t* cand, int64_t n, int64_t ld,
                                   const uint8_t* mask, const float* h_ref, const float* eps, int32_t n_mc,
                                   int32_t q, void* work, int64_t work_bytes, int64_t* h_idx, float* h_val,
                                   int32_t* h_count, float* var_out, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (!L || !state || !h_space || !h_x_obs || !h_y || !h_lengthscale || !h_signal_var || !h_noise_var ||
        !h_ref || !eps || !h_idx || !h_val || !h_count || !work)
        return scoot_fail(ctx, SCOOT_EINVAL, "a required pointer is NULL");
    *h_count = 0;
    if (!scoot_gp_layout_valid(L))
        return scoot_fail(ctx, SCOOT_EINVAL, "GP layout is not one made by scoot_gp_layout_init");
    const int M = L->n_obj;
    if (M < 2 || M > 4) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "fantasy picks need 2 <= M <= 4, got %d", M);
    if (q < 1 || q > SCOOT_MAX_Q) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "q = %d outside 1..%d", q, SCOOT_MAX_Q);
    if (n_mc < 1) return scoot_fail(ctx, SCOOT_EINVAL, "n_mc < 1");
    if ((s = scoot_check_pool(ctx, cand, n, ld, L->d)) != SCOOT_OK) return s;
    if (n > 0x7FFFFFFFll) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "n >= 2^31");
    if (ld_obs < L->n) return scoot_fail(ctx, SCOOT_EINVAL, "ld_obs < n_obs");
    const WorkLayout w = work_layout(L, n, q);
    if (work_bytes < w.bytes)
        return scoot_fail(ctx, SCOOT_EINVAL, "work buffer of %lld bytes, %lld needed", (long long)work_bytes, (long long)w.bytes);
    if ((reinterpret_cast<uintptr_t>(work) & 255u) != 0) return scoot_fail(ctx, SCOOT_EINVAL, "work is not 256-byte aligned");
    if (n == 0) return SCOOT_OK;

    std::vector<HostGP> gps(M);
    for (int m = 0; m < M; ++m) {
        s = scoot_host_gp(h_space, L->d, h_x_obs, ld_obs, L->n, h_y + (size_t)m * L->n, h_lengthscale + (size_t)m * L->d,
                          h_signal_var[m], h_noise_var[m], L->kernel, &gps[m], nullptr);
        if (s != SCOOT_OK) return scoot_fail(ctx, s, "GP of objective %d could not be factored", m);
    }
    {
        // The per-pick downdates rebuild the covariance without warping.  Read
        // after the host factorisation, which overlaps the caller's queued work.
        std::vector<float> scal((size_t)M * 4);
        SCOOT_CUDA(ctx, cudaMemcpy(scal.data(), static_cast<const char*>(state) + L->off_scal,
                                   scal.size() * sizeof(float), cudaMemcpyDeviceToHost));
        for (int m = 0; m < M; ++m)
            if (scal[(size_t)m * 4 + 3] != 0.0f)
                return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "fantasy picks on a warped GP state");
    }
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    char* wk = static_cast<char*>(work);
    FantArgs a;
    std::memset(&a, 0, sizeof(a));
    const unsigned int* n_list = nullptr;
    int64_t n_live = n;
    if (mask) {
        ScootList lst;
        if ((s = scoot_compact(ctx, mask, n, nullptr, 0u, st, &lst)) != SCOOT_OK) return s;
        a.list = lst.list;
        n_list = lst.count;
        unsigned int cnt = 0;
        SCOOT_CUDA(ctx, cudaMemcpyAsync(&cnt, lst.count, 4, cudaMemcpyDeviceToHost, st));
        SCOOT_CUDA(ctx, cudaStreamSynchronize(st));
        n_live = cnt;
    }
    a.n_live = n_live;
    a.ldc = n;
    a.mean = reinterpret_cast<float*>(wk + w.mean);
    a.var = reinterpret_cast<float*>(wk + w.var);
    a.V = reinterpret_cast<float*>(wk + w.V);
    a.C = reinterpret_cast<float*>(wk + w.C);
    a.vp = reinterpret_cast<float*>(wk + w.vp);
    a.cxp = reinterpret_cast<float*>(wk + w.cxp);
    a.inv_s = reinterpret_cast<float*>(wk + w.inv_s);
    a.picked = reinterpret_cast<int64_t*>(wk + w.picked);
    a.n_pad = L->n_rb * 64;
    a.q = q;
    a.acq = reinterpret_cast<float*>(wk + w.acq);
    a.state = static_cast<const char*>(state);
    a.off_fmap = L->off_fmap;
    a.off_ils = L->off_ils;
    a.off_scal = L->off_scal;
    a.n_obs = L->n;
    a.d = L->d;
    a.kernel = L->kernel;
    a.cand = cand;
    a.ld = ld;
    a.box_lo = reinterpret_cast<float*>(wk + w.box_lo);
    a.box_hi = reinterpret_cast<float*>(wk + w.box_hi);
    a.eps = eps;
    a.n_mc = n_mc;
    a.partial = reinterpret_cast<uint64_t*>(wk + w.partial);
    a.best = reinterpret_cast<uint64_t*>(wk + w.best);
    if (n_live > 0) {
        s = scoot_posterior_whitened(ctx, L, state, cand, n, ld, a.list, n_list, reinterpret_cast<float*>(wk + w.mean),
                                     reinterpret_cast<float*>(wk + w.var), reinterpret_cast<float*>(wk + w.V), n, st);
        if (s != SCOOT_OK) return s;
        switch (M) {
        case 2: s = run_picks<2>(ctx, L, a, gps, h_space, cand, ld, h_y, h_ref, q, wk, w, h_idx, h_val, h_count, st); break;
        case 3: s = run_picks<3>(ctx, L, a, gps, h_space, cand, ld, h_y, h_ref, q, wk, w, h_idx, h_val, h_count, st); break;
        default: s = run_picks<4>(ctx, L, a, gps, h_space, cand, ld, h_y, h_ref, q, wk, w, h_idx, h_val, h_count, st); break;
        }
        if (s != SCOOT_OK) return s;
    }
    if (var_out && n_live > 0) {
        int64_t blocks = (n_live + kFThreads - 1) / kFThreads;
        if (blocks > (int64_t)sm_count(ctx->device) * 16) blocks = (int64_t)sm_count(ctx->device) * 16;
        scatter_var<<<(unsigned)blocks, kFThreads, 0, st>>>(a.list, n_live, n, M, a.var, var_out, n);
        SCOOT_LAUNCHED(ctx);
    }
    SCOOT_CUDA(ctx, cudaStreamSynchronize(st));
    return SCOOT_OK;
}

}  // extern "C"
