// Incremental update of the in-edge transpose after a relation update
// (a7, §4.1 cross-chunk relations): instead of re-sorting every edge of the
// store, the old in-edge lists are moved to their new offsets and only the
// new edges are placed, then every in-edge weight is recomputed from its
// logit and its source row's softmax statistics.
//
// Layout facts this relies on (all enforced by the update's preconditions):
//   * the new chunks' rows come after every old row (appends grow the store
//     at the end), so in an old target's list the new sources sort after
//     all old ones;
//   * new chunks have no in-edges before the update and are not linked to
//     each other, so a new chunk's in-edges are exactly its M reciprocal
//     edges;
//   * the out-edge weights are w = exp(aff - max_row) * inv_row with the
//     per-row (max, inv) kept in `rstat`, so recomputing them here gives the
//     same bits as the row softmax.
#include "ak_common.cuh"

namespace ak {

// inc[row of t] += 1 for every forward pair (new chunk -> old chunk t).
__global__ void k_inc_fwd(const int32_t *__restrict__ nbr_ids, int64_t pairs,
                          const int32_t *__restrict__ row_of, unsigned long long *__restrict__ inc) {
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < pairs;
         p += (int64_t)gridDim.x * blockDim.x)
        atomicAdd(&inc[row_of[nbr_ids[p]]], 1ull);
}

// deg[r] = old in-degree + forward additions; new rows get M (reciprocal).
__global__ void k_in_deg_new(const int64_t *__restrict__ in_ptr_old, int64_t n,
                             const int64_t *__restrict__ inc, int64_t *__restrict__ deg) {
    for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n;
         r += (int64_t)gridDim.x * blockDim.x)
        deg[r] = (in_ptr_old[r + 1] - in_ptr_old[r]) + inc[r];
}

__global__ void k_in_deg_recip(const int32_t *__restrict__ row_of, int64_t first, int64_t n_new,
                               int M, int64_t *__restrict__ deg) {
    for (int64_t a = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; a < n_new;
         a += (int64_t)gridDim.x * blockDim.x)
        deg[row_of[first + a]] += M;
}

// Old lists to their new offsets, in order, each edge's weight recomputed
// from its logit and its source's row statistics on the way (a moved edge
// whose source row did not change gets its old weight back bit for bit).
// Edge-parallel (a row-parallel copy would leave one warp copying a hub's
// ~10^5..10^6 edges): chunks of CHUNK_E edges are dealt
// round-robin to the warps; a warp finds the rows of a chunk at once
// (chunk_rows), then issues all of a lane's loads for the chunk before any
// store.
__global__ __launch_bounds__(256) void k_copy_in_edges(
    const int64_t *__restrict__ in_ptr_old, const int32_t *__restrict__ src_old,
    const float *__restrict__ aff_old, int64_t n, int64_t nnz_old,
    const int64_t *__restrict__ in_ptr_new, int32_t *__restrict__ src_new,
    float *__restrict__ aff_new, const float2 *__restrict__ rstat_row,
    float *__restrict__ w_new) {
    __shared__ int rid_s[8][CHUNK_E];
    constexpr int PER = CHUNK_E / 32;
    const int lane = threadIdx.x & 31;
    int *rid = rid_s[threadIdx.x >> 5];
    const int64_t w0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t n_chunks = (nnz_old + CHUNK_E - 1) / CHUNK_E;
    // chunks dealt round-robin to the warps; the lanes find the first rows
    // of a warp's next 32 chunks at once, one binary search each
    int64_t first = 0;
    int i = 0;
    for (int64_t c = w0; c < n_chunks; c += nw, ++i) {
        if ((i & 31) == 0) {
            const int64_t cl = c + (int64_t)lane * nw;
            first = cl < n_chunks ? edge_row(in_ptr_old, n, cl * CHUNK_E) : 0;
        }
        const int64_t base = c * CHUNK_E;
        const int64_t r_lo = __shfl_sync(0xffffffffu, first, i & 31);
        {
            int rows[PER];
            chunk_rows(in_ptr_old, n, nnz_old, base, r_lo, rid, rows);
            int32_t src[PER];
            float a[PER];
            int64_t pos[PER];
#pragma unroll
            for (int j = 0; j < PER; ++j) {
                const int64_t e = base + 32 * j + lane;
                const int64_t row = r_lo + rows[j];
                const bool ok = e < nnz_old;
                src[j] = ok ? src_old[e] : 0;
                a[j] = ok ? aff_old[e] : 0.f;
                pos[j] = ok ? e + (in_ptr_new[row] - in_ptr_old[row]) : -1;
            }
            float2 st[PER];
#pragma unroll
            for (int j = 0; j < PER; ++j) st[j] = pos[j] >= 0 ? rstat_row[src[j]] : make_float2(0.f, 0.f);
#pragma unroll
            for (int j = 0; j < PER; ++j) {
                if (pos[j] < 0) continue;
                src_new[pos[j]] = src[j];
                aff_new[pos[j]] = a[j];
                w_new[pos[j]] = row_softmax_weight(a[j], st[j]);
            }
            __syncwarp();
        }
    }
}

// The row statistics by row: rstat_row[r] = rstat[ext_of[r]] (one gather
// per moved in-edge instead of two).
__global__ void k_rstat_rows(const int32_t *__restrict__ ext_of, const float2 *__restrict__ rstat,
                             int64_t n, float2 *__restrict__ rstat_row) {
    for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n;
         r += (int64_t)gridDim.x * blockDim.x)
        rstat_row[r] = rstat[ext_of[r]];
}

// keys[p] = row of the new chunk of pair p (pairs are [new chunk][slot]).
__global__ void k_pair_src_rows(const int32_t *__restrict__ row_of, int64_t first, int M,
                                int64_t pairs, uint32_t *__restrict__ keys) {
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < pairs;
         p += (int64_t)gridDim.x * blockDim.x)
        keys[p] = (uint32_t)row_of[first + p / M];
}

// Forward edges c -> t, pairs sorted by (row of t, row of c): the i-th
// sorted pair is the (i - fwd_off[row t])-th new source of row t, after the
// row's old list.
__global__ void k_place_fwd(const uint32_t *__restrict__ order, int64_t pairs,
                            const int32_t *__restrict__ nbr_ids, const float *__restrict__ nbr_cos,
                            float scale, int64_t first, int M, const int32_t *__restrict__ row_of,
                            const int64_t *__restrict__ in_ptr_old,
                            const int64_t *__restrict__ in_ptr_new,
                            const int64_t *__restrict__ fwd_off, int32_t *__restrict__ src_new,
                            float *__restrict__ aff_new, const float2 *__restrict__ rstat,
                            float *__restrict__ w_new) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < pairs;
         i += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t p = order[i];
        const int64_t rt = row_of[nbr_ids[p]];
        const int64_t pos = in_ptr_new[rt] + (in_ptr_old[rt + 1] - in_ptr_old[rt]) + (i - fwd_off[rt]);
        const float a = scale * nbr_cos[p];
        src_new[pos] = row_of[first + p / M];
        aff_new[pos] = a;
        w_new[pos] = row_softmax_weight(a, rstat[first + p / M]);   // source: chunk first + p / M
    }
}

// Reciprocal edges t -> c: new chunk c's list holds its M chosen chunks'
// rows in ascending order (rank by counting; one warp per new chunk).
__global__ void k_place_recip(const int32_t *__restrict__ nbr_ids, const float *__restrict__ nbr_cos,
                              float scale, int64_t first, int64_t n_new, int M,
                              const int32_t *__restrict__ row_of,
                              const int64_t *__restrict__ in_ptr_new, int32_t *__restrict__ src_new,
                              float *__restrict__ aff_new, const float2 *__restrict__ rstat,
                              float *__restrict__ w_new) {
    const int lane = threadIdx.x & 31;
    int64_t a = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t stride = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (; a < n_new; a += stride) {
        const int32_t *ids = nbr_ids + a * M;
        const int64_t o = in_ptr_new[row_of[first + a]];
        for (int t = lane; t < M; t += 32) {
            const int32_t rt = row_of[ids[t]];
            int rank = 0;
            for (int u = 0; u < M; ++u) rank += row_of[ids[u]] < rt;
            const float af = scale * nbr_cos[a * M + t];
            src_new[o + rank] = rt;
            aff_new[o + rank] = af;
            w_new[o + rank] = row_softmax_weight(af, rstat[ids[t]]);   // source: chunk ids[t]
        }
    }
}

__global__ void k_in_weights(const int32_t *__restrict__ in_src, const float *__restrict__ in_aff,
                             int64_t nnz, const int32_t *__restrict__ ext_of,
                             const float2 *__restrict__ rstat, float *__restrict__ in_w) {
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < nnz;
         e += (int64_t)gridDim.x * blockDim.x) {
        const float2 s = rstat[ext_of[in_src[e]]];
        in_w[e] = row_softmax_weight(in_aff[e], s);
    }
}

cudaError_t launch_in_weights(const int32_t *in_src, const float *in_aff, int64_t nnz,
                              const int32_t *ext_of, const float2 *rstat, float *in_w,
                              cudaStream_t st) {
    if (nnz <= 0) return cudaSuccess;
    k_in_weights<<<device_sm_count() * 8, 256, 0, st>>>(in_src, in_aff, nnz, ext_of, rstat, in_w);
    return cudaGetLastError();
}

cudaError_t launch_in_edges_update(const InEdgeUpdate &u, const InEdgeScratch &s, cudaStream_t st,
                                   int *launches) {
    const int sms = device_sm_count();
    const int64_t pairs = u.n_new * u.M;
    int L = 0;
    cudaError_t e = cudaMemsetAsync(s.inc, 0, (size_t)(u.n + 1) * 8, st);
    if (e != cudaSuccess) return e;
    if (pairs > 0) {
        k_inc_fwd<<<sms * 4, 256, 0, st>>>(u.nbr_ids, pairs, u.row_of, (unsigned long long *)s.inc);
        ++L;
    }
    k_in_deg_new<<<sms * 4, 256, 0, st>>>(u.in_ptr_old, u.n, s.inc, s.deg);
    ++L;
    if (u.reciprocal && u.n_new > 0) {
        k_in_deg_recip<<<sms, 256, 0, st>>>(u.row_of, u.first, u.n_new, u.M, s.deg);
        ++L;
    }
    e = cudaGetLastError();
    if (e == cudaSuccess) e = scan_exclusive(s.deg, u.in_ptr_new, u.n, s.tmp, s.tmp_bytes, st);
    if (e == cudaSuccess) e = scan_exclusive(s.inc, s.fwd_off, u.n, s.tmp, s.tmp_bytes, st);
    if (e != cudaSuccess) return e;
    const int64_t nnz_old = u.nnz_new - pairs * (u.reciprocal ? 2 : 1);
    if (nnz_old > 0) {
        k_rstat_rows<<<sms * 4, 256, 0, st>>>(u.ext_of, u.rstat, u.n, s.rstat_row);
        const int64_t warps = ceil_div<int64_t>(nnz_old, CHUNK_E);
        const int64_t grid = ceil_div<int64_t>(warps, 8);
        k_copy_in_edges<<<(unsigned)(grid < (int64_t)sms * 6 ? grid : (int64_t)sms * 6), 256, 0,
                          st>>>(u.in_ptr_old, u.in_src_old, u.in_aff_old, u.n, nnz_old,
                                u.in_ptr_new, u.in_src_new, u.in_aff_new, s.rstat_row,
                                u.in_w_new);
        L += 2;
    }
    if (pairs > 0) {
        // forward pairs by (target row, source row): sort by source row,
        // then stably by target row
        k_pair_src_rows<<<sms * 2, 256, 0, st>>>(u.row_of, u.first, u.M, pairs, s.keys);
        e = cudaGetLastError();
        if (e == cudaSuccess) e = launch_iota(s.vals, pairs, st);
        bool alt = false;
        if (e == cudaSuccess)
            e = radix_sort_pairs(s.keys, s.vals, s.keys2, s.vals2, pairs, u.row_bits, s.tmp,
                                 s.tmp_bytes, st, &alt);
        if (e != cudaSuccess) return e;
        uint32_t *k1 = alt ? s.keys2 : s.keys, *v1 = alt ? s.vals2 : s.vals;
        uint32_t *k2 = alt ? s.keys : s.keys2, *v2 = alt ? s.vals : s.vals2;
        e = launch_map_keys(v1, u.nbr_ids, u.row_of, k1, pairs, st);
        bool alt2 = false;
        if (e == cudaSuccess)
            e = radix_sort_pairs(k1, v1, k2, v2, pairs, u.row_bits, s.tmp, s.tmp_bytes, st, &alt2);
        if (e != cudaSuccess) return e;
        k_place_fwd<<<sms * 2, 256, 0, st>>>(alt2 ? v2 : v1, pairs, u.nbr_ids, u.nbr_cos, u.scale,
                                             u.first, u.M, u.row_of, u.in_ptr_old, u.in_ptr_new,
                                             s.fwd_off, u.in_src_new, u.in_aff_new, u.rstat,
                                             u.in_w_new);
        ++L;
        if (u.reciprocal) {
            k_place_recip<<<sms * 2, 256, 0, st>>>(u.nbr_ids, u.nbr_cos, u.scale, u.first, u.n_new,
                                                   u.M, u.row_of, u.in_ptr_new, u.in_src_new,
                                                   u.in_aff_new, u.rstat, u.in_w_new);
            ++L;
        }
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (launches) *launches += L;
    return cudaGetLastError();
}

}  // namespace ak
