// Host-side, synchronous preparation of per-round state (no device work):
//  - the GP state blob: fp64 Cholesky factor of K + tau^2 I, alpha and
//    L^{-1} (Section 4.3), cast to fp32 in the tiled layout the kernels read;
//  - the box decomposition of the region the Pareto front does not dominate
//    (Section 4.4, used by the Monte-Carlo EHVI of Eq. 7);
//  - validation and packing of the random forest of Eq. (3).
#include <algorithm>
#include <cmath>
#include <cstring>
#include <limits>
#include <thread>
#include <vector>

#include "internal.h"

namespace {

constexpr int64_t kAlign = 256;
constexpr int kRowBlock = 64;   // rows of L^{-1} per tile
constexpr int kColChunk = 32;   // columns of L^{-1} per tile
constexpr int kForestChunkNodes = 6144;   // 48 KiB of nodes staged at a time: four forest blocks per SM
constexpr int kMaxPatterns = 4096;        // joint category patterns of the GP's categorical table

int64_t align_up(int64_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

bool is_finite(double x) { return std::isfinite(x); }

// GP states with at least kParallelRows observations are prepared with the
// objectives spread over the library's persistent host threads, and with at
// least kColumnRows with L^{-1}'s columns split kColumnThreads ways per
// objective (below that, handing work to another thread costs more than it
// saves).
constexpr int kParallelRows = 32;
constexpr int kColumnRows = 128;
constexpr int kColumnThreads = 4;
constexpr int kKmatRows = 128;  // K + tau^2 I in kKmatChunks row ranges from this n
constexpr int kKmatChunks = 4;

// sum_k a[k] b[k] for k < len, with four independent partial sums (the fp64
// accumulation chains of the factorisation would otherwise run at FMA latency).
double dot(const double* a, const double* b, int len) {
    double s0 = 0.0, s1 = 0.0, s2 = 0.0, s3 = 0.0;
    int k = 0;
    for (; k + 4 <= len; k += 4) {
        s0 += a[k] * b[k];
        s1 += a[k + 1] * b[k + 1];
        s2 += a[k + 2] * b[k + 2];
        s3 += a[k + 3] * b[k + 3];
    }
    for (; k < len; ++k) s0 += a[k] * b[k];
    return (s0 + s1) + (s2 + s3);
}

double stored_value(const scoot_param& p, uint32_t w) {
    if (p.kind == SCOOT_CONTINUOUS) {
        float f;
        std::memcpy(&f, &w, 4);
        return (double)f;
    }
    return (double)(int32_t)w;
}

// Feature coordinate of a stored value (categoricals keep their index).
double feature(const scoot_param& p, double v) {
    switch (p.kind) {
    case SCOOT_INT_LOG:
        return (std::log(v) - std::log((double)p.lo)) / (std::log((double)p.hi) - std::log((double)p.lo));
    case SCOOT_INT_UNIFORM:
    case SCOOT_CONTINUOUS:
        return p.hi > p.lo ? (v - (double)p.lo) / ((double)p.hi - (double)p.lo) : 0.0;
    default:
        return v;
    }
}

double matern(double r, int kernel) {
    if (kernel == SCOOT_MATERN32) {
        double a = std::sqrt(3.0) * r;
        return (1.0 + a) * std::exp(-a);
    }
    double a = std::sqrt(5.0) * r;
    return (1.0 + a + a * a / 3.0) * std::exp(-a);
}

bool valid_space(const scoot_param* sp, int32_t d) {
    for (int c = 0; c < d; ++c) {
        const scoot_param& p = sp[c];
        if (p.kind == SCOOT_CATEGORICAL) {
            if (p.n_choices < 1) return false;
        } else if (p.kind == SCOOT_INT_LOG) {
            if (!(p.lo > 0.0f) || !(p.hi > p.lo)) return false;
        } else if (p.kind == SCOOT_INT_UNIFORM || p.kind == SCOOT_CONTINUOUS) {
            if (!is_finite(p.lo) || !is_finite(p.hi) || p.hi < p.lo) return false;
        } else {
            return false;
        }
    }
    return true;
}

}  // namespace

double HostGP::cov(const double* ua, const double* ub) const {
    double r2 = 0.0;
    for (int c = 0; c < d; ++c) {
        if (cat[c]) {
            if (ua[c] != ub[c]) r2 += 1.0 / (ell[c] * ell[c]);
        } else {
            const double t = (ua[c] - ub[c]) / ell[c];
            r2 += t * t;
        }
    }
    return sf2 * matern(std::sqrt(r2), kernel);
}

void HostGP::warp_features(double* uf) const {
    if (warp.empty()) return;
    for (int c = 0; c < d; ++c) {
        if (cat[c]) continue;
        const double x = std::min(std::max(uf[c], 0.0), 1.0);
        uf[c] = 1.0 - std::pow(1.0 - std::pow(x, warp[2 * c]), warp[2 * c + 1]);
    }
}

void HostGP::kstar(const double* ux, double* k) const {
    std::vector<double> w(ux, ux + d);
    warp_features(w.data());
    for (int j = 0; j < n; ++j) k[j] = cov(w.data(), &u[(size_t)j * d]);
}

void HostGP::solve_lower(const double* b, double* x) const {
    for (int i = 0; i < n; ++i) {
        double t = b[i];
        t -= dot(&chol[(size_t)i * n], x, i);
        x[i] = t / chol[(size_t)i * n + i];
    }
}

bool scoot_host_features(const scoot_param* sp, int d, const uint32_t* words, int64_t ld, int64_t j, double* u) {
    for (int c = 0; c < d; ++c) {
        const double v = stored_value(sp[c], words[(size_t)c * ld + j]);
        if (!is_finite(v)) return false;
        if (sp[c].kind == SCOOT_INT_LOG && !(v > 0.0)) return false;
        u[c] = feature(sp[c], v);
    }
    return true;
}

scoot_status scoot_host_gp(const scoot_param* sp, int d, const uint32_t* x_obs, int64_t ld_obs, int n,
                           const float* y, const float* lengthscale, float signal_var, float noise_var,
                           int kernel, HostGP* g, double* cond, const float* warp) {
    if (!(signal_var > 0.0f) || !is_finite(signal_var) || !(noise_var >= 0.0f) || !is_finite(noise_var))
        return SCOOT_EINVAL;
    g->n = n;
    g->d = d;
    g->kernel = kernel;
    g->sf2 = signal_var;
    g->tau2 = noise_var;
    g->u.assign((size_t)n * d, 0.0);
    g->cat.assign(d, 0);
    g->ell.assign(d, 1.0);
    g->warp.clear();
    for (int c = 0; c < d; ++c) {
        if (!(lengthscale[c] > 0.0f) || !is_finite(lengthscale[c])) return SCOOT_EINVAL;
        g->ell[c] = lengthscale[c];
        g->cat[c] = sp[c].kind == SCOOT_CATEGORICAL;
    }
    if (warp) {
        g->warp.assign(2 * (size_t)d, 1.0);
        for (int c = 0; c < d; ++c) {
            if (g->cat[c]) continue;
            for (int t = 0; t < 2; ++t) {
                if (!(warp[2 * c + t] > 0.0f) || !is_finite(warp[2 * c + t])) return SCOOT_EINVAL;
                g->warp[2 * c + t] = warp[2 * c + t];
            }
        }
    }
    for (int j = 0; j < n; ++j) {
        if (!is_finite(y[j])) return SCOOT_EINVAL;
        if (!scoot_host_features(sp, d, x_obs, ld_obs, j, &g->u[(size_t)j * d])) return SCOOT_EINVAL;
        g->warp_features(&g->u[(size_t)j * d]);
    }
    // K + tau^2 I from features scaled once (ordinal u / l; categorical
    // mismatches weigh 1 / l^2): the same k(a, b) as HostGP::cov without a
    // division per pair.
    std::vector<double> us((size_t)n * d), icat(d, 0.0);
    for (int c = 0; c < d; ++c)
        if (g->cat[c]) icat[c] = 1.0 / (g->ell[c] * g->ell[c]);
    for (int j = 0; j < n; ++j)
        for (int c = 0; c < d; ++c)
            us[(size_t)j * d + c] = g->cat[c] ? g->u[(size_t)j * d + c] : g->u[(size_t)j * d + c] / g->ell[c];
    std::vector<double>& K = g->chol;
    K.assign((size_t)n * n, 0.0);
    auto rows = [&](int i0, int i1) {
        for (int i = i0; i < i1; ++i) {
            const double* ui = &us[(size_t)i * d];
            for (int j = 0; j <= i; ++j) {
                const double* uj = &us[(size_t)j * d];
                double r2 = 0.0;
                for (int c = 0; c < d; ++c) {
                    const double t = ui[c] - uj[c];
                    r2 += g->cat[c] ? (t != 0.0 ? icat[c] : 0.0) : t * t;
                }
                K[(size_t)i * n + j] = g->sf2 * matern(std::sqrt(r2), g->kernel) + (i == j ? g->tau2 : 0.0);
            }
        }
    };
    if (n >= kKmatRows) {
        // row ranges of equal triangle area: row i has i + 1 entries
        int bounds[kKmatChunks + 1];
        for (int k = 0; k <= kKmatChunks; ++k) bounds[k] = (int)std::lround(n * std::sqrt((double)k / kKmatChunks));
        scoot_host_parallel(kKmatChunks, [&](int k) { rows(bounds[k], bounds[k + 1]); });
    } else {
        rows(0, n);
    }
    double pmin = std::numeric_limits<double>::infinity(), pmax = 0.0;
    for (int j = 0; j < n; ++j) {
        double s = K[(size_t)j * n + j];
        s -= dot(&K[(size_t)j * n], &K[(size_t)j * n], j);
        if (!(s > 0.0) || !is_finite(s)) return SCOOT_EINVAL;
        const double piv = std::sqrt(s);
        K[(size_t)j * n + j] = piv;
        pmin = std::min(pmin, piv);
        pmax = std::max(pmax, piv);
        for (int i = j + 1; i < n; ++i) {
            double t = K[(size_t)i * n + j];
            t -= dot(&K[(size_t)i * n], &K[(size_t)j * n], j);
            K[(size_t)i * n + j] = t / piv;
        }
        for (int i = 0; i < j; ++i) K[(size_t)i * n + j] = 0.0;  // keep the upper triangle zero
    }
    if (cond) *cond = (pmax / pmin) * (pmax / pmin);
    // alpha = C^{-T} C^{-1} y
    std::vector<double> tmp(n), yd(n);
    for (int j = 0; j < n; ++j) yd[j] = y[j];
    g->solve_lower(yd.data(), tmp.data());
    g->alpha.assign(n, 0.0);
    for (int i = n - 1; i >= 0; --i) {
        double t = tmp[i];
        for (int k = i + 1; k < n; ++k) t -= K[(size_t)k * n + i] * g->alpha[k];
        g->alpha[i] = t / K[(size_t)i * n + i];
    }
    return SCOOT_OK;
}

extern "C" {

const char* scoot_status_string(scoot_status s) {
    switch (s) {
    case SCOOT_OK: return "ok";
    case SCOOT_EINVAL: return "invalid argument";
    case SCOOT_ENOMEM: return "out of device memory";
    case SCOOT_ECUDA: return "CUDA runtime error";
    case SCOOT_EDEVICE: return "device-side index or value check failed";
    case SCOOT_ETIMEOUT: return "bounded device wait timed out";
    case SCOOT_EUNSUPPORTED: return "unsupported size or option";
    default: return "unknown status";
    }
}

// ---------------------------------------------------------------- GP state

}  // extern "C"

namespace {

scoot_status gp_layout_compute(int32_t n, int32_t d, int32_t n_obj, int32_t kernel, int32_t n_ord, int32_t n_pat,
                               scoot_gp_layout* out) {
    std::memset(out, 0, sizeof(*out));
    if (n < 1 || d < 1 || n_obj < 1) return SCOOT_EINVAL;
    if (n > SCOOT_MAX_OBS || d > SCOOT_MAX_DIM || n_obj > SCOOT_MAX_OBJ) return SCOOT_EUNSUPPORTED;
    if (kernel != SCOOT_MATERN52 && kernel != SCOOT_MATERN32) return SCOOT_EINVAL;
    if (n_ord < 0 || n_ord > d || n_pat < 1 || n_pat > kMaxPatterns) return SCOOT_EINVAL;
    out->n = n;
    out->d = d;
    out->n_obj = n_obj;
    out->kernel = kernel;
    out->n_rb = (n + kRowBlock - 1) / kRowBlock;
    out->n_tiles = out->n_rb * (out->n_rb + 1);  // row block b spans 2(b+1) column chunks
    out->n_ord = n_ord;
    out->n_pat = n_pat;
    int64_t off = 0;
    out->off_fmap = off;  off = align_up(off + (int64_t)d * 4 * 4);
    out->off_xs = off;    off = align_up(off + (int64_t)n_obj * n * d * 4);
    out->off_ils = off;   off = align_up(off + (int64_t)n_obj * d * 4);
    out->off_alpha = off; off = align_up(off + (int64_t)n_obj * n * 4);
    out->off_linv = off;  off = align_up(off + (int64_t)n_obj * out->n_tiles * kColChunk * kRowBlock * 4);
    out->off_scal = off;  off = align_up(off + (int64_t)n_obj * 4 * 4);
    out->off_cat = off;   off = align_up(off + (int64_t)n_obj * n * n_pat * 4);
    out->off_warp = off;  off = align_up(off + (int64_t)n_obj * d * 2 * 4);
    out->bytes = off;
    return SCOOT_OK;
}

}  // namespace

bool scoot_gp_layout_valid(const scoot_gp_layout* L) {
    if (!L) return false;
    scoot_gp_layout chk;
    if (gp_layout_compute(L->n, L->d, L->n_obj, L->kernel, L->n_ord, L->n_pat, &chk) != SCOOT_OK) return false;
    return std::memcmp(&chk, L, sizeof(chk)) == 0;
}

extern "C" {

scoot_status scoot_gp_layout_init(const scoot_param* h_space, int32_t n, int32_t d, int32_t n_obj, int32_t kernel,
                                  scoot_gp_layout* out) {
    if (!out) return SCOOT_EINVAL;
    std::memset(out, 0, sizeof(*out));
    if (!h_space || d < 1) return SCOOT_EINVAL;
    if (d > SCOOT_MAX_DIM) return SCOOT_EUNSUPPORTED;
    if (!valid_space(h_space, d)) return SCOOT_EINVAL;
    int32_t n_ord = 0;
    int64_t n_pat = 1;
    for (int c = 0; c < d; ++c) {
        if (h_space[c].kind == SCOOT_CATEGORICAL) {
            n_pat *= h_space[c].n_choices;
            if (n_pat > kMaxPatterns) return SCOOT_EUNSUPPORTED;
        } else {
            ++n_ord;
        }
    }
    return gp_layout_compute(n, d, n_obj, kernel, n_ord, (int32_t)n_pat, out);
}

scoot_status scoot_gp_prepare(const scoot_param* h_space, const uint32_t* h_x_obs, int64_t ld_obs,
                              const float* h_y, const float* h_lengthscale,
                              const float* h_signal_var, const float* h_noise_var,
                              const scoot_gp_layout* L, void* h_blob, double* h_cond) {
    return scoot_gp_prepare_warped(h_space, h_x_obs, ld_obs, h_y, h_lengthscale, h_signal_var, h_noise_var,
                                   nullptr, L, h_blob, h_cond);
}

scoot_status scoot_gp_prepare_warped(const scoot_param* h_space, const uint32_t* h_x_obs, int64_t ld_obs,
                                     const float* h_y, const float* h_lengthscale,
                                     const float* h_signal_var, const float* h_noise_var,
                                     const float* h_warp, const scoot_gp_layout* L, void* h_blob,
                                     double* h_cond) {
    if (!h_blob) return SCOOT_EINVAL;
    return scoot_gp_build(h_space, h_x_obs, ld_obs, h_y, h_lengthscale, h_signal_var, h_noise_var, h_warp, L, h_blob,
                          h_cond, nullptr);
}

}  // extern "C"

scoot_status scoot_gp_build(const scoot_param* h_space, const uint32_t* h_x_obs, int64_t ld_obs, const float* h_y,
                            const float* h_lengthscale, const float* h_signal_var, const float* h_noise_var,
                            const float* h_warp, const scoot_gp_layout* L, void* h_blob, double* h_cond,
                            void* h_fant) {
    if (!h_space || !h_x_obs || !h_y || !h_lengthscale || !h_signal_var || !h_noise_var || !L || (!h_blob && !h_fant))
        return SCOOT_EINVAL;
    if (h_fant && h_warp) return SCOOT_EUNSUPPORTED;
    scoot_gp_layout chk;
    if (scoot_gp_layout_init(h_space, L->n, L->d, L->n_obj, L->kernel, &chk) != SCOOT_OK ||
        std::memcmp(&chk, L, sizeof(chk)) != 0)
        return SCOOT_EINVAL;
    const int n = L->n, d = L->d, M = L->n_obj;
    if (ld_obs < n || !valid_space(h_space, d)) return SCOOT_EINVAL;
    for (int m = 0; m < M; ++m) {
        if (!(h_signal_var[m] > 0.0f) || !is_finite(h_signal_var[m])) return SCOOT_EINVAL;
        if (!(h_noise_var[m] >= 0.0f) || !is_finite(h_noise_var[m])) return SCOOT_EINVAL;
        for (int c = 0; c < d; ++c)
            if (!(h_lengthscale[m * d + c] > 0.0f) || !is_finite(h_lengthscale[m * d + c])) return SCOOT_EINVAL;
        for (int j = 0; j < n; ++j)
            if (!is_finite(h_y[m * n + j])) return SCOOT_EINVAL;
    }

    // Without a blob (the fantasy state alone) the fp32 parts are written to
    // a scratch copy that is dropped.
    std::vector<char> scratch;
    if (!h_blob) scratch.resize((size_t)L->bytes);
    char* blob = h_blob ? static_cast<char*>(h_blob) : scratch.data();
    std::memset(blob, 0, (size_t)L->bytes);
    FantHeader* fh = static_cast<FantHeader*>(h_fant);
    char* fbase = static_cast<char*>(h_fant);
    // Feature order: ordinal parameters first, then categorical ones, so the
    // kernels' distance loops need no per-dimension branch on the kind.
    std::vector<int> order;
    for (int c = 0; c < d; ++c)
        if (h_space[c].kind != SCOOT_CATEGORICAL) order.push_back(c);
    for (int c = 0; c < d; ++c)
        if (h_space[c].kind == SCOOT_CATEGORICAL) order.push_back(c);
    float* fmap = reinterpret_cast<float*>(blob + L->off_fmap);
    for (int f = 0; f < d; ++f) {
        const int c = order[f];
        const scoot_param& p = h_space[c];
        float a = 0.f, b = 0.f;
        if (p.kind == SCOOT_INT_LOG) {
            a = (float)std::log((double)p.lo);
            b = (float)(1.0 / (std::log((double)p.hi) - std::log((double)p.lo)));
        } else if (p.kind != SCOOT_CATEGORICAL) {
            a = p.lo;
            b = p.hi > p.lo ? (float)(1.0 / ((double)p.hi - (double)p.lo)) : 0.0f;
        }
        fmap[f * 4 + 0] = (float)p.kind;
        fmap[f * 4 + 1] = a;
        fmap[f * 4 + 2] = b;
        fmap[f * 4 + 3] = (float)c;
    }
    // Categorical features: n_choices and the mixed-radix stride of the pattern id.
    {
        int stride = 1;
        for (int f = L->n_ord; f < d; ++f) {
            const scoot_param& p = h_space[order[f]];
            fmap[f * 4 + 1] = (float)p.n_choices;
            fmap[f * 4 + 2] = (float)stride;
            stride *= p.n_choices;
        }
    }
    float* cat = reinterpret_cast<float*>(blob + L->off_cat);

    float* xs = reinterpret_cast<float*>(blob + L->off_xs);
    float* ils = reinterpret_cast<float*>(blob + L->off_ils);
    float* alpha_out = reinterpret_cast<float*>(blob + L->off_alpha);
    float* linv_out = reinterpret_cast<float*>(blob + L->off_linv);
    float* scal = reinterpret_cast<float*>(blob + L->off_scal);
    float* warp_out = reinterpret_cast<float*>(blob + L->off_warp);

    // One objective's part of the blob; objectives write disjoint parts.
    auto prep = [&](int m) -> scoot_status {
        std::vector<double> Li((size_t)n * n);
        HostGP g;
        scoot_status s = scoot_host_gp(h_space, d, h_x_obs, ld_obs, n, h_y + (size_t)m * n,
                                       h_lengthscale + (size_t)m * d, h_signal_var[m], h_noise_var[m],
                                       L->kernel, &g, h_cond ? &h_cond[m] : nullptr,
                                       h_warp ? h_warp + (size_t)m * d * 2 : nullptr);
        if (s != SCOOT_OK) return s;
        for (int f = 0; f < d; ++f) {
            const int c = order[f];
            warp_out[((size_t)m * d + f) * 2 + 0] = g.warp.empty() || g.cat[c] ? 1.0f : (float)g.warp[2 * c];
            warp_out[((size_t)m * d + f) * 2 + 1] = g.warp.empty() || g.cat[c] ? 1.0f : (float)g.warp[2 * c + 1];
        }
        for (int f = 0; f < d; ++f) {
            const int c = order[f];
            const double l = g.ell[c];
            ils[m * d + f] = g.cat[c] ? (float)(1.0 / (l * l)) : (float)(1.0 / l);
            for (int j = 0; j < n; ++j)
                xs[((size_t)m * n + j) * d + f] = g.cat[c] ? (float)g.u[(size_t)j * d + c]
                                                           : (float)(g.u[(size_t)j * d + c] / l);
        }
        for (int i = 0; i < n; ++i) alpha_out[(size_t)m * n + i] = (float)g.alpha[i];
        if (fh) {  // the fp64 inputs of the fantasy picks' rank-1 terms (original parameter order)
            double* fu = reinterpret_cast<double*>(fbase + fh->off_u);
            double* fell = reinterpret_cast<double*>(fbase + fh->off_ell) + (size_t)m * d;
            double* falpha = reinterpret_cast<double*>(fbase + fh->off_alpha) + (size_t)m * n;
            if (m == 0) std::memcpy(fu, g.u.data(), (size_t)n * d * sizeof(double));
            std::memcpy(fell, g.ell.data(), (size_t)d * sizeof(double));
            std::memcpy(falpha, g.alpha.data(), (size_t)n * sizeof(double));
        }
        // L^{-1}: column by column, C col = e_col; column c is zero above row
        // c, so its forward substitution starts there (n^3 / 6 in all).
        // Li holds the columns contiguously: Li[c * n + i] = L^{-1}[i][c].
        const std::vector<double>& C = g.chol;
        std::fill(Li.begin(), Li.end(), 0.0);
        std::vector<double> rdiag(n);
        for (int i = 0; i < n; ++i) rdiag[i] = 1.0 / C[(size_t)i * n + i];
        auto columns = [&](int c0, int step) {
            for (int c = c0; c < n; c += step) {
                double* col = &Li[(size_t)c * n];
                col[c] = rdiag[c];
                for (int i = c + 1; i < n; ++i) {
                    const double* Ci = &C[(size_t)i * n];
                    col[i] = -dot(Ci + c, col + c, i - c) * rdiag[i];
                }
            }
        };
        // Columns are independent: large states split them over host threads
        // (interleaved, since column c costs ~(n - c)^2 / 2).
        if (n >= kColumnRows) {
            const int t = kColumnThreads;
            scoot_host_parallel(t, [&](int k) { columns(k, t); });
        } else {
            columns(0, 1);
        }
        if (fh) {
            double* flinv = reinterpret_cast<double*>(fbase + fh->off_linv) + (size_t)m * n * n;
            std::memcpy(flinv, Li.data(), (size_t)n * n * sizeof(double));
        }
        // Tiles: row block rb covers rows [64 rb, 64 rb + 64) and column
        // chunks cj = 0 .. 2 rb + 1 of 32 columns; tile[jj][ii] = Li[row][col].
        float* tiles = linv_out + (size_t)m * L->n_tiles * kColChunk * kRowBlock;
        int t = 0;
        for (int rb = 0; rb < L->n_rb; ++rb)
            for (int cj = 0; cj < 2 * (rb + 1); ++cj, ++t)
                for (int jj = 0; jj < kColChunk; ++jj)
                    for (int ii = 0; ii < kRowBlock; ++ii) {
                        const int row = rb * kRowBlock + ii, c = cj * kColChunk + jj;
                        float v = 0.0f;
                        if (row < n && c <= row) v = (float)Li[(size_t)c * n + row];
                        tiles[((size_t)t * kColChunk + jj) * kRowBlock + ii] = v;
                    }
        // Categorical part of r^2 for every (observation, category pattern).
        for (int j = 0; j < n; ++j)
            for (int pat = 0; pat < L->n_pat; ++pat) {
                double r2 = 0.0;
                int rest = pat;
                for (int f = L->n_ord; f < d; ++f) {
                    const int c = order[f];
                    const int v = rest % h_space[c].n_choices;
                    rest /= h_space[c].n_choices;
                    if ((double)v != g.u[(size_t)j * d + c]) r2 += 1.0 / (g.ell[c] * g.ell[c]);
                }
                cat[((size_t)m * n + j) * L->n_pat + pat] = (float)r2;
            }
        float ybest = -std::numeric_limits<float>::infinity();
        for (int j = 0; j < n; ++j) ybest = std::max(ybest, h_y[(size_t)m * n + j]);
        scal[m * 4 + 0] = h_signal_var[m];
        scal[m * 4 + 1] = h_noise_var[m];
        scal[m * 4 + 2] = ybest;
        scal[m * 4 + 3] = h_warp ? 1.0f : 0.0f;
        return SCOOT_OK;
    };
    // Large states: objectives in parallel host threads (the work is O(n^3)
    // per objective; small ones stay on the calling thread).
    std::vector<scoot_status> status(M, SCOOT_OK);
    if (M > 1 && n >= kParallelRows) {
        scoot_host_parallel(M, [&](int m) { status[m] = prep(m); });
    } else {
        for (int m = 0; m < M; ++m) status[m] = prep(m);
    }
    for (int m = 0; m < M; ++m)
        if (status[m] != SCOOT_OK) return status[m];
    return SCOOT_OK;
}

extern "C" {

// ---------------------------------------------------------------- boxes

// The points of y ([M][n_pts]) strictly above the reference point that no
// other such point dominates (duplicates kept once: the first).  False on a
// non-finite value.
static bool pareto_front(const float* h_y, int32_t n_pts, int M, const float* h_ref,
                         std::vector<std::vector<double>>* front) {
    for (int j = 0; j < M; ++j)
        if (!is_finite(h_ref[j])) return false;
    std::vector<std::vector<double>> pts;
    for (int i = 0; i < n_pts; ++i) {
        std::vector<double> p(M);
        bool above = true;
        for (int j = 0; j < M; ++j) {
            p[j] = h_y[(size_t)j * n_pts + i];
            if (!is_finite(p[j])) return false;
            above &= p[j] > (double)h_ref[j];
        }
        if (above) pts.push_back(p);
    }
    front->clear();
    for (size_t i = 0; i < pts.size(); ++i) {
        bool dom = false;
        for (size_t k = 0; k < pts.size() && !dom; ++k) {
            if (k == i) continue;
            bool ge = true, gt = false;
            for (int j = 0; j < M; ++j) {
                ge &= pts[k][j] >= pts[i][j];
                gt |= pts[k][j] > pts[i][j];
            }
            dom = ge && (gt || k < i);
        }
        if (!dom) front->push_back(pts[i]);
    }
    return true;
}

scoot_status scoot_boxes_build(const float* h_y, int32_t n_pts, int32_t n_obj, const float* h_ref,
                               int32_t cap, float* h_lo, float* h_hi, int32_t* n_boxes,
                               int32_t* front_size) {
    if (!h_ref || !n_boxes || cap < 0 || n_pts < 0 || (n_pts > 0 && !h_y)) return SCOOT_EINVAL;
    if (n_obj < 2 || n_obj > SCOOT_MAX_OBJ) return SCOOT_EUNSUPPORTED;
    const int M = n_obj;
    std::vector<std::vector<double>> front;
    if (!pareto_front(h_y, n_pts, M, h_ref, &front)) return SCOOT_EINVAL;
    if (front_size) *front_size = (int32_t)front.size();
    // Grid on axes 0 .. M-2: the reference coordinate and the front's.
    const int G = M - 1;
    std::vector<std::vector<double>> axis(G);
    for (int j = 0; j < G; ++j) {
        axis[j].push_back(h_ref[j]);
        for (auto& p : front) axis[j].push_back(p[j]);
        std::sort(axis[j].begin(), axis[j].end());
        axis[j].erase(std::unique(axis[j].begin(), axis[j].end()), axis[j].end());
    }
    const double inf = std::numeric_limits<double>::infinity();
    // Column over a cell: above h = the highest last-objective value among
    // front points that dominate the cell's upper corner on axes 0..M-2.
    std::vector<int> k(G, 0);
    struct Box { std::vector<double> lo, hi; };
    std::vector<Box> out;
    bool done = false;
    while (!done) {
        // Cells along the last grid axis (G-1) are merged while h is unchanged.
        std::vector<double> up(G);
        for (int j = 0; j < G - 1; ++j)
            up[j] = k[j] + 1 < (int)axis[j].size() ? axis[j][k[j] + 1] : inf;
        const int last = G - 1;
        const int cells = (int)axis[last].size();
        double prev_h = 0.0;
        for (int kk = 0; kk < cells; ++kk) {
            up[last] = kk + 1 < cells ? axis[last][kk + 1] : inf;
            double h = -inf;
            for (auto& p : front) {
                bool dominates = true;
                for (int j = 0; j < G; ++j) dominates &= p[j] >= up[j];
                if (dominates) h = std::max(h, p[M - 1]);
            }
            double lo_last = std::max((double)h_ref[M - 1], h);
            if (kk > 0 && lo_last == prev_h) {
                out.back().hi[last] = up[last];
                continue;
            }
            Box b;
            b.lo.resize(M);
            b.hi.resize(M);
            for (int j = 0; j < G; ++j) {
                b.lo[j] = axis[j][j == last ? kk : k[j]];
                b.hi[j] = up[j];
            }
            b.lo[M - 1] = lo_last;
            b.hi[M - 1] = inf;
            out.push_back(b);
            prev_h = lo_last;
        }
        // Next cell of axes 0 .. G-2 (odometer).
        int j = G - 2;
        while (j >= 0) {
            if (++k[j] < (int)axis[j].size()) break;
            k[j] = 0;
            --j;
        }
        done = j < 0;
    }
    *n_boxes = (int32_t)out.size();
    if ((int32_t)out.size() > cap) return SCOOT_EUNSUPPORTED;
    if (!out.empty() && (!h_lo || !h_hi)) return SCOOT_EINVAL;
    for (size_t b = 0; b < out.size(); ++b)
        for (int j = 0; j < M; ++j) {
            h_lo[b * M + j] = (float)out[b].lo[j];
            h_hi[b * M + j] = std::isinf(out[b].hi[j]) ? std::numeric_limits<float>::infinity()
                                                       : (float)out[b].hi[j];
        }
    return SCOOT_OK;
}

scoot_status scoot_boxes_index(const float* h_lo, const float* h_hi, int32_t n_boxes, int32_t n_obj,
                               int32_t grid_cap, float* h_grid, int32_t* h_n_grid, uint32_t* h_corner) {
    if (n_boxes < 0 || grid_cap < 0 || !h_n_grid) return SCOOT_EINVAL;
    if (n_obj < 2 || n_obj > SCOOT_MAX_OBJ) return SCOOT_EUNSUPPORTED;
    if (n_boxes > 0 && (!h_lo || !h_hi || !h_corner)) return SCOOT_EINVAL;
    const int M = n_obj;
    for (int j = 0; j < M; ++j) {
        std::vector<float> axis;
        for (int b = 0; b < n_boxes; ++b) {
            const float lo = h_lo[(size_t)b * M + j], hi = h_hi[(size_t)b * M + j];
            if (!std::isfinite(lo) || std::isnan(hi) || !(hi > lo)) return SCOOT_EINVAL;
            axis.push_back(lo);
            if (std::isfinite(hi)) axis.push_back(hi);
        }
        std::sort(axis.begin(), axis.end());
        axis.erase(std::unique(axis.begin(), axis.end()), axis.end());
        h_n_grid[j] = (int32_t)axis.size();
        if ((int64_t)axis.size() > grid_cap || axis.size() > 65535) return SCOOT_EUNSUPPORTED;
        if (!axis.empty() && !h_grid) return SCOOT_EINVAL;
        std::copy(axis.begin(), axis.end(), h_grid + (size_t)j * grid_cap);
        auto index = [&](float v) -> uint32_t {
            if (std::isinf(v)) return (uint32_t)axis.size();
            return (uint32_t)(std::lower_bound(axis.begin(), axis.end(), v) - axis.begin());
        };
        for (int b = 0; b < n_boxes; ++b)
            h_corner[(size_t)b * M + j] = index(h_lo[(size_t)b * M + j]) | (index(h_hi[(size_t)b * M + j]) << 16);
    }
    return SCOOT_OK;
}

// ---------------------------------------------------------------- forest

scoot_status scoot_forest_layout_init(const scoot_node* h_nodes, const int32_t* h_tree_offset,
                                      int32_t n_trees, int32_t d, int32_t leaf_scale,
                                      scoot_forest_layout* out) {
    if (!out) return SCOOT_EINVAL;
    std::memset(out, 0, sizeof(*out));
    if (!h_nodes || !h_tree_offset || n_trees < 1 || d < 1 || d > SCOOT_MAX_DIM || leaf_scale < 1)
        return SCOOT_EINVAL;
    if (h_tree_offset[0] != 0) return SCOOT_EINVAL;
    int max_depth = 0;
    std::vector<int> depth;
    std::vector<int32_t> chunks;  // first tree, count, first node, node count
    int chunk_first = 0, chunk_nodes = 0;
    for (int t = 0; t < n_trees; ++t) {
        int32_t b = h_tree_offset[t], e = h_tree_offset[t + 1];
        int size = e - b;
        if (size < 1 || size > 65535) return SCOOT_EINVAL;
        if (size > kForestChunkNodes) return SCOOT_EUNSUPPORTED;
        depth.assign(size, -1);
        depth[0] = 0;
        for (int i = 0; i < size; ++i) {
            const scoot_node& nd = h_nodes[b + i];
            if (depth[i] < 0) return SCOOT_EINVAL;  // unreachable node
            if (nd.flags & 1) {
                float v = nd.val;
                if (!(v >= 0.0f) || v > (float)leaf_scale || v != std::floor(v)) return SCOOT_EINVAL;
                max_depth = std::max(max_depth, depth[i]);
            } else {
                if (nd.feat >= d || !is_finite(nd.val)) return SCOOT_EINVAL;
                int l = nd.left;
                if (l <= i || l + 1 >= size) return SCOOT_EINVAL;
                if (depth[l] >= 0 || depth[l + 1] >= 0) return SCOOT_EINVAL;  // shared child
                depth[l] = depth[l + 1] = depth[i] + 1;
            }
        }
        if (chunk_nodes + size > kForestChunkNodes) {
            chunks.insert(chunks.end(), {chunk_first, t - chunk_first, h_tree_offset[chunk_first], chunk_nodes});
            chunk_first = t;
            chunk_nodes = 0;
        }
        chunk_nodes += size;
    }
    chunks.insert(chunks.end(), {chunk_first, n_trees - chunk_first, h_tree_offset[chunk_first], chunk_nodes});
    out->n_trees = n_trees;
    out->n_nodes = h_tree_offset[n_trees];
    out->d = d;
    out->leaf_scale = leaf_scale;
    out->max_depth = max_depth;
    out->n_chunks = (int32_t)(chunks.size() / 4);
    for (size_t c = 0; c < chunks.size(); c += 4)
        out->max_chunk_nodes = std::max(out->max_chunk_nodes, chunks[c + 3]);
    int64_t off = 0;
    out->off_chunks = off; off = align_up(off + (int64_t)out->n_chunks * 16);
    out->off_roots = off;  off = align_up(off + (int64_t)n_trees * 4);
    out->off_nodes = off;  off = align_up(off + (int64_t)out->n_nodes * 8);
    out->bytes = off;
    return SCOOT_OK;
}

scoot_status scoot_forest_pack(const scoot_forest_layout* L, const scoot_node* h_nodes,
                               const int32_t* h_tree_offset, void* h_blob) {
    if (!L || !h_nodes || !h_tree_offset || !h_blob) return SCOOT_EINVAL;
    scoot_forest_layout chk;
    scoot_status s = scoot_forest_layout_init(h_nodes, h_tree_offset, L->n_trees, L->d, L->leaf_scale, &chk);
    if (s != SCOOT_OK) return s;
    if (std::memcmp(&chk, L, sizeof(chk)) != 0) return SCOOT_EINVAL;
    char* blob = static_cast<char*>(h_blob);
    std::memset(blob, 0, (size_t)L->bytes);
    int32_t* ch = reinterpret_cast<int32_t*>(blob + L->off_chunks);
    int c = 0, first = 0, nodes = 0;
    for (int t = 0; t < L->n_trees; ++t) {
        int size = h_tree_offset[t + 1] - h_tree_offset[t];
        if (nodes + size > kForestChunkNodes) {
            ch[c * 4 + 0] = first; ch[c * 4 + 1] = t - first;
            ch[c * 4 + 2] = h_tree_offset[first]; ch[c * 4 + 3] = nodes;
            ++c; first = t; nodes = 0;
        }
        nodes += size;
    }
    ch[c * 4 + 0] = first; ch[c * 4 + 1] = L->n_trees - first;
    ch[c * 4 + 2] = h_tree_offset[first]; ch[c * 4 + 3] = nodes;
    std::memcpy(blob + L->off_roots, h_tree_offset, (size_t)L->n_trees * 4);
    // Nodes with the left child counted from the first node of the node's
    // chunk, so a walk in shared memory needs no per-tree offset.
    scoot_node* out = reinterpret_cast<scoot_node*>(blob + L->off_nodes);
    for (int k = 0; k < L->n_chunks; ++k) {
        const int first = ch[k * 4 + 0], count = ch[k * 4 + 1], node0 = ch[k * 4 + 2];
        for (int t = first; t < first + count; ++t)
            for (int i = h_tree_offset[t]; i < h_tree_offset[t + 1]; ++i) {
                out[i] = h_nodes[i];
                if (!(h_nodes[i].flags & 1))
                    out[i].left = (uint16_t)(h_tree_offset[t] - node0 + h_nodes[i].left);
            }
    }
    return SCOOT_OK;
}

}  // extern "C"

// ---------------------------------------------------------------- fantasy state

void scoot_fant_layout(int32_t n, int32_t d, int32_t M, int32_t q, FantHeader* h) {
    std::memset(h, 0, sizeof(*h));
    h->magic = kFantMagic;
    h->n = n;
    h->d = d;
    h->M = M;
    h->q = q;
    int64_t off = align_up((int64_t)sizeof(FantHeader));
    h->off_space = off; off = align_up(off + (int64_t)d * 4 * 8);
    h->off_u = off;     off = align_up(off + (int64_t)n * d * 8);
    h->off_ell = off;   off = align_up(off + (int64_t)M * d * 8);
    h->off_alpha = off; off = align_up(off + (int64_t)M * n * 8);
    h->off_linv = off;  off = align_up(off + (int64_t)M * n * n * 8);
    h->off_front = off; off = align_up(off + (int64_t)n * M * 8);
    h->bytes = off;
}

scoot_status scoot_fant_header(const scoot_param* h_space, const scoot_gp_layout* L, const float* h_y,
                               const float* h_signal_var, const float* h_noise_var, const float* h_ref, int32_t q,
                               void* h_fant, int64_t cap) {
    if (!h_space || !L || !h_y || !h_signal_var || !h_noise_var || !h_ref || !h_fant) return SCOOT_EINVAL;
    const int n = L->n, d = L->d, M = L->n_obj;
    if (M < 2 || M > SCOOT_MAX_OBJ) return SCOOT_EUNSUPPORTED;
    if (q < 1 || q > SCOOT_MAX_Q) return SCOOT_EUNSUPPORTED;
    FantHeader h;
    scoot_fant_layout(n, d, M, q, &h);
    if (cap < h.bytes) return SCOOT_ENOMEM;
    std::vector<std::vector<double>> front;
    if (!pareto_front(h_y, n, M, h_ref, &front)) return SCOOT_EINVAL;
    h.kernel = L->kernel;
    h.front0 = (int32_t)front.size();
    h.front_cap = h.front0 + q;
    // Cells of the box decomposition of a front of front_cap points: at most
    // front_cap + 1 grid coordinates on each of the first M - 1 axes.
    double cells = 1.0;
    for (int j = 0; j < M - 1; ++j) cells *= (double)(h.front_cap + 1);
    h.box_cap = cells > (double)kFantBoxMax ? kFantBoxMax : (int32_t)cells;
    for (int m = 0; m < M; ++m) {
        h.ref[m] = h_ref[m];
        h.sf2[m] = h_signal_var[m];
        h.tau2[m] = h_noise_var[m];
    }
    char* base = static_cast<char*>(h_fant);
    std::memcpy(base, &h, sizeof(h));
    double* sp = reinterpret_cast<double*>(base + h.off_space);
    for (int c = 0; c < d; ++c) {
        sp[c * 4 + 0] = h_space[c].kind;
        sp[c * 4 + 1] = h_space[c].lo;
        sp[c * 4 + 2] = h_space[c].hi;
        sp[c * 4 + 3] = h_space[c].n_choices;
    }
    double* fr = reinterpret_cast<double*>(base + h.off_front);
    for (size_t i = 0; i < front.size(); ++i)
        for (int m = 0; m < M; ++m) fr[i * M + m] = front[i][m];
    return SCOOT_OK;
}

extern "C" {

scoot_status scoot_fantasy_state_bytes(const scoot_gp_layout* L, int32_t q, int64_t* bytes) {
    if (!L || !bytes || !scoot_gp_layout_valid(L)) return SCOOT_EINVAL;
    if (q < 1 || q > SCOOT_MAX_Q) return SCOOT_EUNSUPPORTED;
    FantHeader h;
    scoot_fant_layout(L->n, L->d, L->n_obj, q, &h);
    *bytes = h.bytes;
    return SCOOT_OK;
}

scoot_status scoot_fantasy_prepare(const scoot_param* h_space, const scoot_gp_layout* L, const uint32_t* h_x_obs,
                                   int64_t ld_obs, const float* h_y, const float* h_lengthscale,
                                   const float* h_signal_var, const float* h_noise_var, const float* h_ref,
                                   int32_t q, void* h_out, int64_t cap, int32_t* box_cap) {
    if (!L || !scoot_gp_layout_valid(L)) return SCOOT_EINVAL;
    scoot_status s = scoot_fant_header(h_space, L, h_y, h_signal_var, h_noise_var, h_ref, q, h_out, cap);
    if (s != SCOOT_OK) return s;
    s = scoot_gp_build(h_space, h_x_obs, ld_obs, h_y, h_lengthscale, h_signal_var, h_noise_var, nullptr, L,
                       nullptr, nullptr, h_out);
    if (s != SCOOT_OK) return s;
    if (box_cap) *box_cap = static_cast<const FantHeader*>(h_out)->box_cap;
    return SCOOT_OK;
}

}  // extern "C"
