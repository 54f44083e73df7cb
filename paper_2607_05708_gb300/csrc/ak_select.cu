// Top-k selection (a3) with score normalisation by Z (a1) and the page
// resolve + distinct-page count (a4): the top-p selection and FetchByID of
// query-aware retrieval (arXiv 2607.05708, §4.1, Algorithm 1) and the
// locality gap |P(R_t)| (§3.2).
#include "ak_common.cuh"

namespace ak {

constexpr int SEL_THREADS = 256;

// SIGNED=false: non-negative scores (retrieval); SIGNED=true: any finite
// value (cosines of the relation update).  Either way a larger key is a
// better candidate and equal values prefer the lower chunk ID.
template <bool SIGNED>
__device__ __forceinline__ unsigned long long sel_key(float v, uint32_t id) {
    const uint32_t hi = SIGNED ? ordered_bits(v) : __float_as_uint(v);
    return ((unsigned long long)hi << 32) | (unsigned long long)(~id);
}
template <bool SIGNED>
__device__ __forceinline__ float sel_value(unsigned long long key) {
    const uint32_t hi = (uint32_t)(key >> 32);
    return SIGNED ? unordered_bits(hi) : __uint_as_float(hi);
}

// Candidate pass.  Thread (r, c) of CTA g scans rows g*rows_per_cta + r,
// + lanes, ... for query column c and keeps its k best keys in a sorted
// list in shared memory (slot-major, so a warp's accesses are contiguous).
// Reads of a row by the CTA's threads are contiguous, hence coalesced.
template <bool SIGNED>
__global__ __launch_bounds__(SEL_THREADS) void k_topk_candidates(
    const float *__restrict__ s, int64_t n, int bp, int lanes, int k, int64_t rows_per_cta,
    const int32_t *__restrict__ ext_of, int64_t id_limit, unsigned long long *__restrict__ cand) {
    extern __shared__ unsigned long long lists[];   // [k][SEL_THREADS]
    const int tid = threadIdx.x;
    const int c = tid % bp, r = tid / bp;
    const bool active = r < lanes;
    for (int i = 0; i < k; ++i) lists[i * SEL_THREADS + tid] = 0ull;
    unsigned long long kth = 0ull;
    if (active) {
        const int64_t r0 = (int64_t)blockIdx.x * rows_per_cta;
        const int64_t r1 = r0 + rows_per_cta < n ? r0 + rows_per_cta : n;
        constexpr int U = 8;   // rows in flight per thread
        for (int64_t j0 = r0 + r; j0 < r1; j0 += (int64_t)U * lanes) {
            float v[U];
            int32_t id[U];
#pragma unroll
            for (int q = 0; q < U; ++q) {
                const int64_t j = j0 + (int64_t)q * lanes;
                v[q] = j < r1 ? s[j * bp + c] : 0.f;
                id[q] = j < r1 ? ext_of[j] : 0;
            }
#pragma unroll
            for (int q = 0; q < U; ++q) {
                const int64_t j = j0 + (int64_t)q * lanes;
                if (j >= r1) break;
                if ((int64_t)id[q] >= id_limit) continue;
                const unsigned long long key = sel_key<SIGNED>(v[q], (uint32_t)id[q]);
                if (key > kth) {
                    int i = k - 1;
                    while (i > 0 && lists[(i - 1) * SEL_THREADS + tid] < key) {
                        lists[i * SEL_THREADS + tid] = lists[(i - 1) * SEL_THREADS + tid];
                        --i;
                    }
                    lists[i * SEL_THREADS + tid] = key;
                    kth = lists[(k - 1) * SEL_THREADS + tid];
                }
            }
        }
        const int64_t list = (int64_t)blockIdx.x * lanes + r;
        unsigned long long *dst = cand + (list * bp + c) * k;
        for (int i = 0; i < k; ++i) dst[i] = lists[i * SEL_THREADS + tid];
    }
}

// Exact k-th largest key of column c among all candidate lists by an
// MSB-first radix select (8 bits a pass); the k winners are left in win[]
// (unordered) and their count in *win_n.  Keys are unique (each row is seen
// by one list only) and lists pad with key 0, below every real key.
__device__ void radix_select_column(const unsigned long long *__restrict__ cand, int64_t lists,
                                    int bp, int k, int c, unsigned long long *win, int *win_n,
                                    int *hist, unsigned long long *s_prefix, int *s_remaining) {
    const int tid = threadIdx.x;
    const int64_t total = lists * (int64_t)k;
    if (tid == 0) {
        *s_prefix = 0ull;
        *s_remaining = k;
        *win_n = 0;
    }
    __syncthreads();
    unsigned long long pmask = 0ull;
    for (int pass = 0; pass < 8; ++pass) {
        const int sh = 56 - 8 * pass;
        hist[tid] = 0;
        __syncthreads();
        const unsigned long long prefix = *s_prefix;
        for (int64_t i = tid; i < total; i += SEL_THREADS) {
            const int64_t l = i / k, slot = i % k;
            const unsigned long long key = cand[(l * bp + c) * k + slot];
            if ((key & pmask) == prefix) atomicAdd(&hist[(key >> sh) & 0xff], 1);
        }
        __syncthreads();
        if (tid == 0) {
            int rem = *s_remaining, cum = 0, sel = 0;
            for (int d = 255; d >= 0; --d) {
                if (cum + hist[d] >= rem) {
                    sel = d;
                    break;
                }
                cum += hist[d];
            }
            *s_remaining = rem - cum;
            *s_prefix = prefix | ((unsigned long long)sel << sh);
        }
        pmask |= 0xffull << sh;
        __syncthreads();
    }
    const unsigned long long kth = *s_prefix;
    for (int64_t i = tid; i < total; i += SEL_THREADS) {
        const int64_t l = i / k, slot = i % k;
        const unsigned long long key = cand[(l * bp + c) * k + slot];
        if (key >= kth && key != 0ull) {
            int p = atomicAdd(win_n, 1);
            if (p < 64) win[p] = key;
        }
    }
    __syncthreads();
}

// Retrieval merge, one CTA per real query column: the k winners ordered by
// key (score desc, id asc), normalised by Z = sum of the score pass's tile
// partials, resolved to pages, and their distinct pages counted.
__global__ __launch_bounds__(SEL_THREADS) void k_topk_merge(
    const unsigned long long *__restrict__ cand, int64_t lists, int bp, int k,
    const float *__restrict__ zpart, int64_t n_ztiles, const int32_t *__restrict__ row_of,
    const int32_t *__restrict__ page_row, int64_t *__restrict__ ids, float *__restrict__ scores,
    int32_t *__restrict__ page_ids, int32_t *__restrict__ n_pages, int *status) {
    __shared__ int hist[256];
    __shared__ unsigned long long s_prefix;
    __shared__ int s_remaining;
    __shared__ unsigned long long win[64];
    __shared__ int win_n;
    __shared__ double zred[SEL_THREADS / 32];
    __shared__ int pg[64];
    const int c = blockIdx.x;
    const int tid = threadIdx.x;
    double z = 0.0;
    for (int64_t t = tid; t < n_ztiles; t += SEL_THREADS) z += (double)zpart[t * bp + c];
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    if ((tid & 31) == 0) zred[tid >> 5] = z;
    radix_select_column(cand, lists, bp, k, c, win, &win_n, hist, &s_prefix, &s_remaining);
    if (tid == 0 && win_n != k) set_status(status, AKASHIC_EDEVICE);
    const int got = win_n < k ? win_n : k;
    if (tid < got) {
        const unsigned long long key = win[tid];
        int rank = 0;
        for (int t = 0; t < got; ++t) rank += win[t] > key;
        double zsum = 0.0;
        for (int w = 0; w < SEL_THREADS / 32; ++w) zsum += zred[w];
        const uint32_t id = key_id(key);
        const int64_t o = (int64_t)c * k + rank;
        ids[o] = (int64_t)id;
        scores[o] = (float)((double)sel_value<false>(key) / zsum);
        const int32_t p = page_row ? page_row[row_of[id]] : 0;
        pg[rank] = p;
        if (page_ids) page_ids[o] = p;
    }
    __syncthreads();
    if (n_pages && tid < 32) {
        int distinct = 0;
        for (int a = tid; a < got; a += 32) {
            bool first = true;
            for (int b2 = 0; b2 < a; ++b2) first &= pg[b2] != pg[a];
            distinct += first;
        }
        for (int o = 16; o > 0; o >>= 1) distinct += __shfl_xor_sync(0xffffffffu, distinct, o);
        if (tid == 0) n_pages[c] = distinct;
    }
}

// Relation-update merge: the M best prior chunks of new chunk c (ordered by
// cosine desc, id asc) into nbr_ids / nbr_cos rows c_base + c.
__global__ __launch_bounds__(SEL_THREADS) void k_topm_merge(
    const unsigned long long *__restrict__ cand, int64_t lists, int bp, int k, int64_t c_base,
    int32_t *__restrict__ nbr_ids, float *__restrict__ nbr_cos, int *status) {
    __shared__ int hist[256];
    __shared__ unsigned long long s_prefix;
    __shared__ int s_remaining;
    __shared__ unsigned long long win[64];
    __shared__ int win_n;
    const int c = blockIdx.x;
    const int tid = threadIdx.x;
    radix_select_column(cand, lists, bp, k, c, win, &win_n, hist, &s_prefix, &s_remaining);
    if (tid == 0 && win_n != k) set_status(status, AKASHIC_EDEVICE);
    const int got = win_n < k ? win_n : k;
    if (tid < got) {
        const unsigned long long key = win[tid];
        int rank = 0;
        for (int t = 0; t < got; ++t) rank += win[t] > key;
        const int64_t o = (c_base + c) * k + rank;
        nbr_ids[o] = (int32_t)key_id(key);
        nbr_cos[o] = sel_value<true>(key);
    }
}

SelectPlan select_plan(int64_t n, int bp, int k, int sm_count) {
    SelectPlan sp;
    sp.lanes = SEL_THREADS / bp > 0 ? SEL_THREADS / bp : 1;
    // at least ~4k rows per list, at most two CTAs per SM
    int64_t want = ceil_div<int64_t>(n, (int64_t)sp.lanes * 4 * k);
    int64_t cap = 2 * (int64_t)sm_count;
    sp.grid = (int)(want < 1 ? 1 : (want > cap ? cap : want));
    sp.lists = (int64_t)sp.grid * sp.lanes;
    return sp;
}

cudaError_t launch_select(const SelectPlan &sp, const float *s, int64_t n, int bp, int b, int k,
                          unsigned long long *cand, const float *zpart, int64_t n_ztiles,
                          const int32_t *ext_of, const int32_t *row_of, const int32_t *page_row,
                          int64_t *ids, float *scores, int32_t *page_ids, int32_t *n_pages,
                          int *status, cudaStream_t st, int *launches) {
    const size_t smem = (size_t)k * SEL_THREADS * sizeof(unsigned long long);
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev]) {
        const int mx = 64 * SEL_THREADS * (int)sizeof(unsigned long long);
        cudaError_t e = cudaFuncSetAttribute(k_topk_candidates<false>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(k_topk_candidates<true>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
        if (e != cudaSuccess) return e;
        attr_set[dev] = true;
    }
    const int64_t rows_per_cta = ceil_div<int64_t>(n, sp.grid);
    k_topk_candidates<false><<<sp.grid, SEL_THREADS, smem, st>>>(
        s, n, bp, sp.lanes, k, rows_per_cta, ext_of, (int64_t)1 << 40, cand);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_topk_merge<<<b, SEL_THREADS, 0, st>>>(cand, sp.lists, bp, k, zpart, n_ztiles, row_of,
                                            page_row, ids, scores, page_ids, n_pages, status);
    if (launches) *launches += 2;
    return cudaGetLastError();
}

cudaError_t launch_select_signed(const SelectPlan &sp, const float *s, int64_t n, int bp, int b,
                                 int k, unsigned long long *cand, const int32_t *ext_of,
                                 int64_t id_limit, int64_t c_base, int32_t *nbr_ids,
                                 float *nbr_cos, int *status, cudaStream_t st, int *launches) {
    const size_t smem = (size_t)k * SEL_THREADS * sizeof(unsigned long long);
    cudaError_t e = cudaFuncSetAttribute(k_topk_candidates<true>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         64 * SEL_THREADS * (int)sizeof(unsigned long long));
    if (e != cudaSuccess) return e;
    const int64_t rows_per_cta = ceil_div<int64_t>(n, sp.grid);
    k_topk_candidates<true><<<sp.grid, SEL_THREADS, smem, st>>>(s, n, bp, sp.lanes, k,
                                                                rows_per_cta, ext_of, id_limit,
                                                                cand);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_topm_merge<<<b, SEL_THREADS, 0, st>>>(cand, sp.lists, bp, k, c_base, nbr_ids, nbr_cos,
                                            status);
    if (launches) *launches += 2;
    return cudaGetLastError();
}

}  // namespace ak
