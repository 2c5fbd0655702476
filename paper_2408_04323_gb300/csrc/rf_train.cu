// Training of the feasibility forest (Algorithm 1's TRAIN: random forest
// regression of the crash labels, Section 4.6), one regression tree per
// block on a bootstrap sample given by the caller.
//
// CART with squared error, grown breadth first: a node with m samples and p
// positive labels has SSE p (m - p) / m; it becomes a leaf at the depth
// limit, when pure, or when no split separates its samples; otherwise it
// takes the split "x_f <= v" (v one of its samples' values of feature f, not
// the largest) with the smallest SSE(left) + SSE(right).  Labels are 0/1, so
// the comparison is exact in integers: SSE(left) + SSE(right) =
// (p_l (m_l - p_l) m_r + p_r (m_r - p_r) m_l) / (m_l m_r), compared by cross
// multiplication; ties go to the lower feature, then the lower value.  A leaf
// stores round(V p / m) votes (halves up).  Breadth-first numbering puts the
// two children of a node next to each other, after it.

#include "internal.h"

namespace {

constexpr int kTrainThreads = 256;
constexpr int kTrainWarps = kTrainThreads / 32;

struct Split {
    long long num, den;  // SSE(left) + SSE(right) = num / den; den = 0: none
    int f, nl, pl;
    float v;
};

__device__ __forceinline__ bool better(const Split& a, const Split& b) {
    if (a.den == 0) return false;
    if (b.den == 0) return true;
    const long long l = a.num * b.den, r = b.num * a.den;
    if (l != r) return l < r;
    if (a.f != b.f) return a.f < b.f;
    return a.v < b.v;
}

__device__ __forceinline__ Split shfl_split(const Split& s, int o) {
    Split t;
    t.num = __shfl_xor_sync(0xffffffffu, s.num, o);
    t.den = __shfl_xor_sync(0xffffffffu, s.den, o);
    t.f = __shfl_xor_sync(0xffffffffu, s.f, o);
    t.nl = __shfl_xor_sync(0xffffffffu, s.nl, o);
    t.pl = __shfl_xor_sync(0xffffffffu, s.pl, o);
    t.v = __shfl_xor_sync(0xffffffffu, s.v, o);
    return t;
}

__device__ __forceinline__ float feature_value(const uint32_t* obs, int64_t ld, uint32_t float_cols, int f, int i) {
    const uint32_t w = obs[(int64_t)f * ld + i];
    return ((float_cols >> f) & 1u) ? __uint_as_float(w) : (float)(int32_t)w;
}

// A total order on float bit patterns (numeric order on finite values, -0
// before +0), so that the ranks below form a permutation even when a value
// is NaN (such observations are rejected by the training kernel).
__device__ __forceinline__ uint32_t order_key(float x) {
    const uint32_t u = __float_as_uint(x);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// perm[f][r] = the observation of rank r in feature f (ties by index): one
// thread per (observation, feature).
__global__ void __launch_bounds__(kTrainThreads)
rank_kernel(const uint32_t* __restrict__ obs, int64_t ld, uint32_t float_cols, int n, uint16_t* __restrict__ perm) {
    const int i = blockIdx.x * kTrainThreads + threadIdx.x, f = blockIdx.y;
    if (i >= n) return;
    const uint32_t ki = order_key(feature_value(obs, ld, float_cols, f, i));
    int r = 0;
    for (int j = 0; j < n; ++j) {
        const uint32_t kj = order_key(feature_value(obs, ld, float_cols, f, j));
        r += kj < ki || (kj == ki && j < i);
    }
    perm[f * n + r] = (uint16_t)i;
}

// One block grows tree blockIdx.x.  Each feature f keeps the bootstrap's
// samples as a list of observation ids sorted by x[f] (a sample drawn c
// times appears c times); the lists are partitioned by node, so the samples
// of a node occupy the same range [b, e) of every list, its left child's
// first, and stay sorted.  A node at depth D reads the lists of buffer D & 1
// and writes its children's into buffer (D + 1) & 1 (the two ranges belong
// to no pending node).  The split search of a list is one prefix sum of the
// labels: at the last position k of a run of equal values, "x[f] <= x_k"
// sends the k - b + 1 samples before it left.
// obs: the observations' words [d][ld] (float_cols: bit f set for a
// continuous parameter f; the others convert from int32); y: labels; boot:
// [T][m] sample indices; perm: [d][n] from rank_kernel; out: [T][ld_nodes]
// nodes, of which tree t writes the first n_out[t] (<= node_cap = 2 m - 1).
__global__ void __launch_bounds__(kTrainThreads)
rf_train_kernel(const uint32_t* __restrict__ obs, int64_t ld, uint32_t float_cols, const uint8_t* __restrict__ y,
                int n, int d, const int32_t* __restrict__ boot, int m, const uint16_t* __restrict__ perm,
                int max_depth, int leaf_scale, int node_cap, int ld_nodes, scoot_node* __restrict__ out,
                int32_t* __restrict__ n_out, uint32_t* __restrict__ err) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    float* col = reinterpret_cast<float*>(smem_raw);                      // [d][n] feature values
    unsigned int* mult = reinterpret_cast<unsigned int*>(col + (size_t)d * n);  // [n] draws of each observation
    uint16_t* ids = reinterpret_cast<uint16_t*>(mult + n);                // [2][d][m] sorted lists
    uint16_t* qb = ids + (size_t)2 * d * m;                               // [node_cap] range begin
    uint16_t* qe = qb + node_cap;                                         // [node_cap] range end
    uint16_t* qp = qe + node_cap;                                         // [node_cap] positives
    uint8_t* qd = reinterpret_cast<uint8_t*>(qp + node_cap);              // [node_cap] depth
    uint8_t* lab = qd + node_cap;                                         // [n] labels
    uint8_t* goleft = lab + n;                                            // [n] side of the current split
    __shared__ Split wbest[2][kTrainWarps];
    __shared__ int wcount[kTrainWarps];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const unsigned int lt = (1u << lane) - 1u;
    const int tree = blockIdx.x;
    scoot_node* nodes = out + (size_t)tree * ld_nodes;

    for (int k = tid; k < n * d; k += kTrainThreads) {
        const int f = k / n, i = k - f * n;
        col[k] = feature_value(obs, ld, float_cols, f, i);
    }
    for (int i = tid; i < n; i += kTrainThreads) {
        lab[i] = y[i];
        mult[i] = 0;
    }
    __syncthreads();
    // draws per observation; only drawn observations are validated
    int bad_value = 0, bad_index = 0;
    for (int k = tid; k < m; k += kTrainThreads) {
        const int32_t i = boot[(size_t)tree * m + k];
        if (i < 0 || i >= n) {
            bad_index = 1;
            continue;
        }
        atomicAdd(mult + i, 1u);
        bad_value |= lab[i] > 1;
        for (int f = 0; f < d; ++f) bad_value |= !isfinite(col[f * n + i]);
    }
    bad_value = __syncthreads_or(bad_value);
    bad_index = __syncthreads_or(bad_index);
    if (bad_value || bad_index) {  // the same in every thread
        if (tid == 0) {
            atomicOr(err, (bad_value ? SCOOT_DEVERR_VALUE : 0u) | (bad_index ? SCOOT_DEVERR_INDEX : 0u));
            n_out[tree] = 0;
        }
        return;
    }
    // root lists: observations in rank order, each repeated by its draws
    for (int f = warp; f < d; f += kTrainWarps) {
        uint16_t* L = ids + f * m;
        int carry = 0;
        for (int r0 = 0; r0 < n; r0 += 32) {
            const int r = r0 + lane;
            int i = 0, c = 0;
            if (r < n) {
                i = perm[f * n + r];
                if (i >= n) i = 0;  // perm is a permutation; kept in range regardless
                c = (int)mult[i];
            }
            int sc = c;
            for (int o = 1; o < 32; o <<= 1) {
                const int t = __shfl_up_sync(0xffffffffu, sc, o);
                if (lane >= o) sc += t;
            }
            const int start = carry + sc - c;
            for (int j = 0; j < c && start + j < m; ++j) L[start + j] = (uint16_t)i;
            carry += __shfl_sync(0xffffffffu, sc, 31);
        }
    }
    {
        int p = 0;
        for (int i = tid; i < n; i += kTrainThreads) p += lab[i] * (int)mult[i];
        for (int o = 16; o > 0; o >>= 1) p += __shfl_xor_sync(0xffffffffu, p, o);
        if (lane == 0) wcount[warp] = p;
        __syncthreads();
        if (tid == 0) {
            int t = 0;
            for (int w = 0; w < kTrainWarps; ++w) t += wcount[w];
            qb[0] = 0;
            qe[0] = (uint16_t)m;
            qp[0] = (uint16_t)t;
            qd[0] = 0;
        }
        __syncthreads();
    }
    int tail = 1;      // queue length, the same in every thread
    int searches = 0;  // split searches so far; selects the wbest buffer
    for (int head = 0; head < tail; ++head) {
        const int b = qb[head], e = qe[head], p = qp[head], depth = qd[head], mn = e - b;
        const uint16_t* src = ids + (size_t)(depth & 1) * d * m;
        Split best{0, 0, 0, 0, 0, 0.0f};
        if (depth < max_depth && p > 0 && p < mn) {  // the same in every thread
            for (int f = warp; f < d; f += kTrainWarps) {
                const uint16_t* L = src + f * m;
                const float* cf = col + f * n;
                int carry = 0;
                for (int k0 = b; k0 < e; k0 += 32) {
                    const int k = k0 + lane;
                    float x = 0.0f;
                    int l = 0;
                    if (k < e) {
                        const int i = L[k];
                        x = cf[i];
                        l = lab[i];
                    }
                    int sc = l;
                    for (int o = 1; o < 32; o <<= 1) {
                        const int t = __shfl_up_sync(0xffffffffu, sc, o);
                        if (lane >= o) sc += t;
                    }
                    const int pl = carry + sc;
                    carry += __shfl_sync(0xffffffffu, sc, 31);
                    if (k < e - 1 && x != cf[L[k + 1]]) {
                        const int nl = k - b + 1, nr = mn - nl, pr = p - pl;
                        const Split cand{(long long)pl * (nl - pl) * nr + (long long)pr * (nr - pr) * nl,
                                         (long long)nl * nr, f, nl, pl, x};
                        if (better(cand, best)) best = cand;
                    }
                }
            }
            for (int o = 16; o > 0; o >>= 1) {
                const Split t = shfl_split(best, o);
                if (better(t, best)) best = t;
            }
            // Alternate buffers: the next write to this one follows the
            // barrier of the next search, which every thread reaches only
            // after reading this one.
            Split* wb = wbest[searches++ & 1];
            if (lane == 0) wb[warp] = best;
            __syncthreads();
            best = wb[0];
            for (int w = 1; w < kTrainWarps; ++w)
                if (better(wb[w], best)) best = wb[w];
        }
        if (best.den != 0 && tail + 2 <= node_cap) {
            const int nl = best.nl;
            // the first nl samples of the split feature's list go left
            const uint16_t* Lf = src + best.f * m;
            for (int k = b + tid; k < e; k += kTrainThreads) goleft[Lf[k]] = k < b + nl;
            __syncthreads();
            uint16_t* dst = ids + (size_t)((depth + 1) & 1) * d * m;
            for (int g = warp; g < d; g += kTrainWarps) {
                const uint16_t* L = src + g * m;
                uint16_t* D = dst + g * m;
                int before = 0;  // left samples before the chunk
                for (int k0 = b; k0 < e; k0 += 32) {
                    const int k = k0 + lane;
                    const int i = k < e ? L[k] : 0;
                    const bool left = k < e && goleft[i];
                    const unsigned int bal = __ballot_sync(0xffffffffu, left);
                    const int lrank = before + __popc(bal & lt);
                    if (k < e) D[left ? b + lrank : b + nl + (k - b - lrank)] = (uint16_t)i;
                    before += __popc(bal);
                }
            }
            if (tid == 0) {
                qb[tail] = (uint16_t)b;
                qe[tail] = (uint16_t)(b + nl);
                qp[tail] = (uint16_t)best.pl;
                qd[tail] = (uint8_t)(depth + 1);
                qb[tail + 1] = (uint16_t)(b + nl);
                qe[tail + 1] = (uint16_t)e;
                qp[tail + 1] = (uint16_t)(p - best.pl);
                qd[tail + 1] = (uint8_t)(depth + 1);
                scoot_node nd;
                nd.val = best.v == 0.0f ? 0.0f : best.v;  // a zero threshold is stored as +0
                nd.left = (uint16_t)tail;
                nd.feat = (uint8_t)best.f;
                nd.flags = 0;
                nodes[head] = nd;
            }
            tail += 2;
            __syncthreads();  // lists and queue entries visible to every thread
        } else if (tid == 0) {
            if (best.den != 0) atomicOr(err, SCOOT_DEVERR_INDEX);  // node capacity exhausted
            scoot_node nd;
            nd.val = (float)((2LL * leaf_scale * p + mn) / (2LL * mn));
            nd.left = 0;
            nd.feat = 0;
            nd.flags = 1;
            nodes[head] = nd;
        }
    }
    if (tid == 0) n_out[tree] = tail;
}

}  // namespace

extern "C" {

scoot_status scoot_rf_train_work_bytes(int32_t n, int32_t d, int64_t* bytes) {
    if (!bytes || n < 1 || d < 1) return SCOOT_EINVAL;
    *bytes = (2 * (int64_t)d * n + 15) / 16 * 16;
    return SCOOT_OK;
}

scoot_status scoot_rf_train(scoot_ctx* ctx, const scoot_param* h_space, int32_t d, const uint32_t* obs, int32_t n,
                            int64_t ld, const uint8_t* labels, const int32_t* boot, int32_t n_trees, int32_t m,
                            int32_t max_depth, int32_t leaf_scale, scoot_node* nodes, int32_t node_cap,
                            int32_t* n_nodes, void* work, int64_t work_bytes, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (n < 1 || n > SCOOT_RF_TRAIN_MAX_OBS)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "n = %d outside 1..%d", n, SCOOT_RF_TRAIN_MAX_OBS);
    if (m < 1 || m > SCOOT_RF_TRAIN_MAX_OBS)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "m = %d outside 1..%d", m, SCOOT_RF_TRAIN_MAX_OBS);
    if (d < 1 || d > SCOOT_MAX_DIM) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "d = %d outside 1..%d", d, SCOOT_MAX_DIM);
    if (n_trees < 0) return scoot_fail(ctx, SCOOT_EINVAL, "n_trees < 0");
    if (max_depth < 0 || max_depth > 255) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "max_depth = %d outside 0..255", max_depth);
    if (leaf_scale < 1 || leaf_scale > (1 << 24))
        return scoot_fail(ctx, SCOOT_EINVAL, "leaf_scale = %d outside 1..2^24", leaf_scale);
    if (node_cap < 2 * m - 1) return scoot_fail(ctx, SCOOT_EINVAL, "node_cap = %d < 2 m - 1 = %d", node_cap, 2 * m - 1);
    if (!h_space) return scoot_fail(ctx, SCOOT_EINVAL, "h_space is NULL");
    if (ld < n) return scoot_fail(ctx, SCOOT_EINVAL, "ld = %lld < n = %d", (long long)ld, n);
    uint32_t float_cols = 0;
    for (int c = 0; c < d; ++c)
        if (h_space[c].kind == SCOOT_CONTINUOUS) float_cols |= 1u << c;
    if (n_trees == 0) return SCOOT_OK;
    if (!obs || !labels || !boot || !nodes || !n_nodes)
        return scoot_fail(ctx, SCOOT_EINVAL, "obs, labels, boot, nodes or n_nodes is NULL");
    const int cap = 2 * m - 1;  // a binary tree over m samples with non-empty leaves has at most 2 m - 1 nodes
    const size_t smem = (size_t)d * n * sizeof(float) + (size_t)n * sizeof(unsigned int) +
                        (size_t)2 * d * m * sizeof(uint16_t) + (size_t)cap * (3 * sizeof(uint16_t) + 1) + (size_t)2 * n;
    static_assert(sizeof(scoot_node) == 8, "scoot_node is 8 bytes");
    if (!work || work_bytes < (int64_t)d * n * (int64_t)sizeof(uint16_t) || !scoot_aligned16(work))
        return scoot_fail(ctx, SCOOT_EINVAL, "work needs %lld bytes, 16-byte aligned", (long long)d * n * 2);
    uint16_t* perm = static_cast<uint16_t*>(work);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    SCOOT_CUDA(ctx, cudaFuncSetAttribute(rf_train_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    rank_kernel<<<dim3((n + kTrainThreads - 1) / kTrainThreads, d), kTrainThreads, 0, st>>>(obs, ld, float_cols, n,
                                                                                          perm);
    SCOOT_LAUNCHED(ctx);
    rf_train_kernel<<<n_trees, kTrainThreads, smem, st>>>(obs, ld, float_cols, labels, n, d, boot, m, perm,
                                                          max_depth, leaf_scale, cap, node_cap, nodes, n_nodes,
                                                          ctx->d_err);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

}  // extern "C"
