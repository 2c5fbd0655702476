// Known-constraint pruning (Eq. 2) and random-forest probability of
// feasibility (Eq. 3) over a structure-of-arrays candidate pool.
#include <cstring>

#include "internal.h"

namespace {

constexpr int kPruneThreads = 256;
constexpr int kRfThreads = 256;
constexpr int kRfCand = 32;                      // candidates per tile (one per lane)
constexpr int kRfGroups = kRfThreads / kRfCand;  // warps = tree groups

struct PruneArgs {
    int32_t n_clauses;
    int32_t exact64;              // 1: every clause sum fits in int64 (sum of |coef| < 2^32)
    scoot_clause cl[SCOOT_MAX_CLAUSES];
};

// Block-wide sum of per-thread counts, added once per block to *count.
__device__ __forceinline__ void add_count(unsigned long long* count, uint32_t mine) {
    __shared__ uint32_t warp_sums[32];
    for (int o = 16; o > 0; o >>= 1) mine += __shfl_xor_sync(0xffffffffu, mine, o);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) warp_sums[warp] = mine;
    __syncthreads();
    if (warp == 0) {
        uint32_t v = lane < (int)(blockDim.x >> 5) ? warp_sums[lane] : 0u;
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0 && v) atomicAdd(count, (unsigned long long)v);
    }
}

// Four consecutive candidates per thread: each clause column is read as one
// 16-byte vector (columns are 16-byte aligned and ld % 4 == 0, so the vector
// at i0 = 4k stays inside the column even for the last, ragged group), every
// guard and term of every clause is loaded without a branch on the guards
// (repeated columns hit L1) so all loads of a group are in flight together,
// the clause sums are exact (int64 when the host has shown that no clause sum
// can overflow it, i.e. sum of |coef| < 2^32 with 32-bit values, else int128),
// and the four mask bytes are stored as one 32-bit word (bytes of a ragged
// tail, or of a mask that is not 4-byte aligned, one by one).
template <bool kExact64>
__device__ __forceinline__ void clause_sums(const scoot_clause& C, const uint32_t* __restrict__ cand, int64_t ld,
                                            int64_t i0, bool (&ok)[4]) {
    bool g[4] = {true, true, true, true};
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        if (k < C.n_guard) {
            const uint4 v = __ldg(reinterpret_cast<const uint4*>(cand + (int64_t)C.guard_param[k] * ld + i0));
            const int32_t want = C.guard_value[k];
            g[0] &= (int32_t)v.x == want;
            g[1] &= (int32_t)v.y == want;
            g[2] &= (int32_t)v.z == want;
            g[3] &= (int32_t)v.w == want;
        }
    }
    if (kExact64) {
        int64_t sum[4] = {0, 0, 0, 0};
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            if (t < C.n_term) {
                const uint4 v = __ldg(reinterpret_cast<const uint4*>(cand + (int64_t)C.term_param[t] * ld + i0));
                const int64_t a = C.coef[t];
                sum[0] += a * (int64_t)(int32_t)v.x;
                sum[1] += a * (int64_t)(int32_t)v.y;
                sum[2] += a * (int64_t)(int32_t)v.z;
                sum[3] += a * (int64_t)(int32_t)v.w;
            }
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) ok[e] &= !g[e] || sum[e] >= C.rhs;
    } else {
        __int128 sum[4] = {0, 0, 0, 0};
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            if (t < C.n_term) {
                const uint4 v = __ldg(reinterpret_cast<const uint4*>(cand + (int64_t)C.term_param[t] * ld + i0));
                const __int128 a = C.coef[t];
                sum[0] += a * (int32_t)v.x;
                sum[1] += a * (int32_t)v.y;
                sum[2] += a * (int32_t)v.z;
                sum[3] += a * (int32_t)v.w;
            }
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) ok[e] &= !g[e] || sum[e] >= (__int128)C.rhs;
    }
}

template <bool kExact64>
__global__ void __launch_bounds__(kPruneThreads)
prune_kernel(const __grid_constant__ PruneArgs a, const uint32_t* __restrict__ cand, int64_t n,
             int64_t ld, uint8_t* __restrict__ mask, unsigned long long* count, int mask_aligned) {
    uint32_t feasible = 0;
    const int64_t groups = (n + 3) / 4;
    for (int64_t gi = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; gi < groups;
         gi += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i0 = 4 * gi;
        bool ok[4] = {true, true, true, true};
        for (int c = 0; c < a.n_clauses; ++c) clause_sums<kExact64>(a.cl[c], cand, ld, i0, ok);
        if (i0 + 4 <= n && mask_aligned) {
            const uint32_t word = (uint32_t)ok[0] | ((uint32_t)ok[1] << 8) | ((uint32_t)ok[2] << 16) |
                                  ((uint32_t)ok[3] << 24);
            *reinterpret_cast<uint32_t*>(mask + i0) = word;
            feasible += (uint32_t)ok[0] + ok[1] + ok[2] + ok[3];
        } else {
            for (int e = 0; e < 4 && i0 + e < n; ++e) {
                mask[i0 + e] = ok[e];
                feasible += ok[e];
            }
        }
    }
    if (count) add_count(count, feasible);
}

struct RfArgs {
    const char* forest;
    int64_t off_chunks, off_roots, off_nodes;
    int32_t n_chunks, n_trees, max_depth, d;
    uint32_t float_cols;          // bit c set: column c holds float32 values
    uint32_t delta_num, delta_den, leaf_scale;
    const uint32_t* cand;
    int64_t n, ld;
    uint32_t* votes;
    uint8_t* mask;
    unsigned long long* count;
    uint32_t* err;
    const int32_t* list;          // live candidates (NULL: all of 0 .. n-1)
    const unsigned int* n_list;
    int32_t max_chunk_nodes;
};

// Persistent blocks of 256 threads score tiles of 32 candidates: lane l of
// warp g serves candidate slot l and walks trees g, g + 8, g + 16, ... of the
// forest, so the 32 lanes of a warp walk the same tree for 32 candidates
// (the upper levels are broadcast loads) and each candidate has eight
// independent walks in flight.  The forest (or one chunk of whole trees at a
// time) sits in shared memory with chunk-relative child indices; the tile's
// feature values sit in shared memory as feat[slot][f] with an odd row
// stride (conflict-free when a warp reads one feature).  The eight partial
// vote counts of a candidate are added through shared memory.
__global__ void __launch_bounds__(kRfThreads)
rf_kernel(const __grid_constant__ RfArgs a) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int fs = a.d | 1;                                                       // odd row stride
    uint2* snodes = reinterpret_cast<uint2*>(smem_raw);                           // chunk nodes
    float* sfeat = reinterpret_cast<float*>(snodes + a.max_chunk_nodes);          // [kRfCand][fs]
    uint32_t* svote = reinterpret_cast<uint32_t*>(sfeat + kRfCand * fs);          // [kRfGroups][kRfCand]
    int32_t* sroot = reinterpret_cast<int32_t*>(svote + kRfGroups * kRfCand);      // [n_trees]

    const int32_t* chunks = reinterpret_cast<const int32_t*>(a.forest + a.off_chunks);
    const int32_t* roots = reinterpret_cast<const int32_t*>(a.forest + a.off_roots);
    const uint2* gnodes = reinterpret_cast<const uint2*>(a.forest + a.off_nodes);
    const int tid = threadIdx.x;
    const int slot = tid & (kRfCand - 1), grp = tid / kRfCand;
    const int64_t n_work = a.list ? (int64_t)*a.n_list : a.n;
    const int64_t n_tiles = (n_work + kRfCand - 1) / kRfCand;
    uint32_t feasible = 0;

    // Staged node word: x = threshold bits (split) or vote count as a float
    // (leaf); y = chunk-relative left child in bits 0..15, the feature's byte
    // offset in a feature row in bits 16..30, bit 31 set for a leaf.
    auto stage_chunk = [&](int ch) {
        const int t0 = chunks[ch * 4 + 0], nt = chunks[ch * 4 + 1];
        const int first_node = chunks[ch * 4 + 2], count = chunks[ch * 4 + 3];
        for (int k = tid; k < count; k += kRfThreads) {
            const uint2 g = __ldg(gnodes + first_node + k);
            const uint32_t leaf = (g.y >> 24) & 1u, feat = (g.y >> 16) & 0xffu;
            snodes[k] = make_uint2(g.x, leaf ? 0x80000000u : ((feat * 4u) << 16) | (g.y & 0xffffu));
        }
        for (int k = tid; k < nt; k += kRfThreads) sroot[t0 + k] = roots[t0 + k] - first_node;
    };
    // Chunk-major: the block walks all of its tiles with chunk 0 of the
    // forest, then all of them with chunk 1, ..., carrying each candidate's
    // partial vote count in votes[] between chunks (the tiles of a block are
    // the same in every chunk), so that a chunk of <= 48 KiB lets four
    // blocks share an SM.
    for (int ch = 0; ch < a.n_chunks; ++ch) {
        const bool first = ch == 0, last = ch + 1 == a.n_chunks;
        __syncthreads();  // the previous chunk's nodes are no longer read
        stage_chunk(ch);  // visible after the first barrier below
        const int t0 = chunks[ch * 4 + 0], nt = chunks[ch * 4 + 1];
        for (int64_t tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
            const int64_t base = tile * kRfCand;
            __syncthreads();  // the previous tile's features and votes are no longer read
            for (int k = tid; k < kRfCand * a.d; k += kRfThreads) {
                const int f = k / kRfCand, c = k - f * kRfCand;
                const int64_t pos = base + c;
                float x = 0.0f;
                if (pos < n_work) {
                    const int64_t i = a.list ? (int64_t)a.list[pos] : pos;
                    const uint32_t w = __ldg(a.cand + (int64_t)f * a.ld + i);
                    x = ((a.float_cols >> f) & 1u) ? __uint_as_float(w) : (float)(int32_t)w;
                }
                sfeat[c * fs + f] = x;
            }
            __syncthreads();
            const int64_t pos = base + slot;
            const bool live = pos < n_work;
            const char* my = reinterpret_cast<const char*>(sfeat + slot * fs);
            uint32_t vote = 0;
            // The lanes of a warp walk the same tree (for 32 candidates) in
            // lockstep, so the upper levels of the tree are broadcast loads;
            // letting each lane run on to its next tree as soon as it reaches
            // a leaf was measured twice as slow: the lanes drift onto
            // different trees and the node loads stop being broadcasts.
            for (int t = t0 + grp; t < t0 + nt && live; t += kRfGroups) {
                int node = sroot[t];
                bool done = false;
#pragma unroll 2
                for (int step = 0; step <= a.max_depth; ++step) {
                    const uint2 nd = snodes[node];
                    if ((int)nd.y < 0) {
                        vote += (uint32_t)__uint_as_float(nd.x);
                        done = true;
                        break;
                    }
                    const float x = *reinterpret_cast<const float*>(my + (nd.y >> 16));
                    node = (int)(nd.y & 0xffffu) + (x <= __uint_as_float(nd.x) ? 0 : 1);
                }
                if (!done) atomicOr(a.err, SCOOT_DEVERR_INDEX);  // deeper than the validated depth
            }
            svote[grp * kRfCand + slot] = vote;
            __syncthreads();
            if (grp == 0 && live) {
                uint32_t v = 0;
#pragma unroll
                for (int g = 0; g < kRfGroups; ++g) v += svote[g * kRfCand + slot];
                const int64_t i = a.list ? (int64_t)a.list[pos] : pos;
                if (!first) v += a.votes[i];  // the earlier chunks' count (written by this thread)
                a.votes[i] = v;
                if (last) {
                    const unsigned __int128 need = (unsigned __int128)a.delta_num * a.leaf_scale * (uint32_t)a.n_trees;
                    const bool ok = (unsigned __int128)a.delta_den * v >= need;
                    if (a.mask) a.mask[i] = ok;
                    feasible += ok;
                }
            }
        }
    }
    if (a.count) add_count(a.count, feasible);
}

int sm_count(int device) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, device);
    return v > 0 ? v : 1;
}

}  // namespace

extern "C" {

scoot_status scoot_prune(scoot_ctx* ctx, const scoot_param* h_space, int32_t d,
                         const scoot_clause* h_clauses, int32_t n_clauses,
                         const uint32_t* cand, int64_t n, int64_t ld,
                         uint8_t* mask, int64_t* n_feasible, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (!h_space) return scoot_fail(ctx, SCOOT_EINVAL, "h_space is NULL");
    if ((s = scoot_check_pool(ctx, cand, n, ld, d)) != SCOOT_OK) return s;
    if (n_clauses < 0 || n_clauses > SCOOT_MAX_CLAUSES)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "n_clauses = %d outside 0..%d", n_clauses, SCOOT_MAX_CLAUSES);
    if (n_clauses > 0 && !h_clauses) return scoot_fail(ctx, SCOOT_EINVAL, "h_clauses is NULL");
    if (n > 0 && !mask) return scoot_fail(ctx, SCOOT_EINVAL, "mask is NULL");
    PruneArgs a;
    std::memset(&a, 0, sizeof(a));
    a.n_clauses = n_clauses;
    for (int c = 0; c < n_clauses; ++c) {
        const scoot_clause& C = h_clauses[c];
        if (C.n_guard < 0 || C.n_guard > 2 || C.n_term < 0 || C.n_term > 4)
            return scoot_fail(ctx, SCOOT_EINVAL, "clause %d: n_guard %d / n_term %d out of range", c, C.n_guard, C.n_term);
        for (int g = 0; g < C.n_guard; ++g) {
            int p = C.guard_param[g];
            if (p < 0 || p >= d || h_space[p].kind == SCOOT_CONTINUOUS)
                return scoot_fail(ctx, SCOOT_EINVAL, "clause %d: guard parameter %d invalid", c, p);
        }
        for (int t = 0; t < C.n_term; ++t) {
            int p = C.term_param[t];
            if (p < 0 || p >= d || h_space[p].kind == SCOOT_CONTINUOUS)
                return scoot_fail(ctx, SCOOT_EINVAL, "clause %d: term parameter %d invalid", c, p);
        }
        a.cl[c] = C;
    }
    unsigned __int128 abs_sum_max = 0;
    for (int c = 0; c < n_clauses; ++c) {
        const scoot_clause& C = h_clauses[c];
        unsigned __int128 abs_sum = 0;
        for (int t = 0; t < C.n_term; ++t)
            abs_sum += (unsigned __int128)(C.coef[t] < 0 ? -(__int128)C.coef[t] : (__int128)C.coef[t]);
        if (abs_sum > abs_sum_max) abs_sum_max = abs_sum;
    }
    a.exact64 = abs_sum_max < ((unsigned __int128)1 << 32);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (n_feasible) SCOOT_CUDA(ctx, cudaMemsetAsync(n_feasible, 0, sizeof(int64_t), st));
    if (n == 0) return SCOOT_OK;
    const int mask_aligned = (reinterpret_cast<uintptr_t>(mask) & 3u) == 0;
    const int64_t groups = (n + 3) / 4;
    int64_t blocks = (groups + kPruneThreads - 1) / kPruneThreads;
    const int64_t cap = (int64_t)sm_count(ctx->device) * 8;
    if (blocks > cap) blocks = cap;
    auto kern = a.exact64 ? prune_kernel<true> : prune_kernel<false>;
    kern<<<(unsigned)blocks, kPruneThreads, 0, st>>>(a, cand, n, ld, mask,
                                                     reinterpret_cast<unsigned long long*>(n_feasible), mask_aligned);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

scoot_status scoot_rf_predict(scoot_ctx* ctx, const scoot_forest_layout* L, const void* forest,
                              const scoot_param* h_space, const uint32_t* cand, int64_t n, int64_t ld,
                              uint32_t delta_num, uint32_t delta_den, uint32_t* votes, uint8_t* mask,
                              int64_t* n_feasible, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (!L || !forest || !h_space) return scoot_fail(ctx, SCOOT_EINVAL, "layout, forest or h_space is NULL");
    if ((s = scoot_check_pool(ctx, cand, n, ld, L->d)) != SCOOT_OK) return s;
    if (L->n_trees < 1 || L->n_chunks < 1 || L->max_depth < 0 || L->leaf_scale < 1)
        return scoot_fail(ctx, SCOOT_EINVAL, "forest layout is not initialised");
    if (delta_den == 0) return scoot_fail(ctx, SCOOT_EINVAL, "delta_den = 0");
    if (n > 0 && !votes) return scoot_fail(ctx, SCOOT_EINVAL, "votes is NULL");
    if (!scoot_aligned16(forest)) return scoot_fail(ctx, SCOOT_EINVAL, "forest blob is not 16-byte aligned");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (n_feasible) SCOOT_CUDA(ctx, cudaMemsetAsync(n_feasible, 0, sizeof(int64_t), st));
    if (n == 0) return SCOOT_OK;

    const int max_chunk_nodes = L->max_chunk_nodes;
    if (max_chunk_nodes < 1 || max_chunk_nodes > L->n_nodes)
        return scoot_fail(ctx, SCOOT_EINVAL, "forest layout is not initialised");
    RfArgs a;
    std::memset(&a, 0, sizeof(a));
    a.forest = static_cast<const char*>(forest);
    a.off_chunks = L->off_chunks;
    a.off_roots = L->off_roots;
    a.off_nodes = L->off_nodes;
    a.n_chunks = L->n_chunks;
    a.n_trees = L->n_trees;
    a.max_depth = L->max_depth;
    a.d = L->d;
    for (int c = 0; c < L->d; ++c)
        if (h_space[c].kind == SCOOT_CONTINUOUS) a.float_cols |= 1u << c;
    a.delta_num = delta_num;
    a.delta_den = delta_den;
    a.leaf_scale = (uint32_t)L->leaf_scale;
    a.cand = cand;
    a.n = n;
    a.ld = ld;
    a.votes = votes;
    a.mask = mask;
    a.count = reinterpret_cast<unsigned long long*>(n_feasible);
    a.err = ctx->d_err;
    if (mask) {
        // Walk only the candidates still in play; the others get 0 votes.
        ScootList lst;
        if ((s = scoot_compact(ctx, mask, n, votes, 0u, st, &lst)) != SCOOT_OK) return s;
        a.list = lst.list;
        a.n_list = lst.count;
    }
    a.max_chunk_nodes = max_chunk_nodes;
    const size_t smem = (size_t)max_chunk_nodes * 8 + (size_t)kRfCand * (L->d | 1) * 4 +
                        (size_t)kRfGroups * kRfCand * 4 + (size_t)L->n_trees * 4;
    SCOOT_CUDA(ctx, cudaFuncSetAttribute(rf_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    int per_sm = 0;
    SCOOT_CUDA(ctx, cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, rf_kernel, kRfThreads, smem));
    if (per_sm < 1) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "forest chunk does not fit in shared memory");
    const int64_t tiles = (n + kRfCand - 1) / kRfCand;
    int64_t blocks = (int64_t)sm_count(ctx->device) * per_sm;
    if (blocks > tiles) blocks = tiles;
    rf_kernel<<<(unsigned)blocks, kRfThreads, smem, st>>>(a);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

}  // extern "C"
