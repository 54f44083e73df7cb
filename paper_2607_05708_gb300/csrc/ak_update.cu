// Relation update (a6, a7): for new chunks, the top-M related prior chunks
// by cosine of the stored embeddings, then the reciprocal insertion of those
// edges into the relation graph's CSR (arXiv 2607.05708, §4.1: cross-chunk
// inference selects the related prior chunks of each new chunk; Algorithm 1's
// LLMSelect of related prior chunks, in its Dense-only form of §5.5).
#include "ak_update.cuh"

namespace ak {

// Gather the embeddings of chunks c0 .. c0+b-1 (rows row_of[c]) into a
// zero-padded bp-row block.
__global__ void k_gather_rows(const uint16_t *__restrict__ emb, const int32_t *__restrict__ row_of,
                              int64_t c0, int b, int bp, int dim, uint16_t *__restrict__ dst) {
    const int64_t total = (int64_t)bp * dim;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / dim, t = i % dim;
        dst[i] = r < b ? emb[(int64_t)row_of[c0 + r] * dim + t] : (uint16_t)0;
    }
}

__global__ void k_ext_sample(const int32_t *__restrict__ ext_of, int64_t n_sample, int64_t stride,
                             int32_t *__restrict__ out) {
    for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < n_sample;
         v += (int64_t)gridDim.x * blockDim.x)
        out[v] = ext_of[v * stride];
}

cudaError_t launch_ext_sample(const int32_t *ext_of, int64_t n_sample, int64_t stride,
                              int32_t *out, cudaStream_t st) {
    if (n_sample <= 0) return cudaSuccess;
    k_ext_sample<<<device_sm_count(), 256, 0, st>>>(ext_of, n_sample, stride, out);
    return cudaGetLastError();
}

// Exact path, batch by batch: dots of every row against 256 new chunks
// written to a slab, then the three-pass selection (used when a fused
// filter buffer overflows).
static akashic_status_t relate_top_m_batched(const UpdateArgs &a, cudaStream_t st, int *launches) {
    const int64_t n_old = a.n_rows;
    int bp_max = 32;
    while (bp_max < 256 && bp_max < a.n_new) bp_max <<= 1;
    int64_t words = 0;
    for (int bp = 32; bp <= bp_max; bp <<= 1) {
        SelectPlan sp = select_plan(n_old, bp, a.M, device_sm_count());
        words = sp.words > words ? sp.words : words;
    }
    uint16_t *qp = (uint16_t *)a.get(SCR_QP, (size_t)bp_max * a.dim * 2);
    float *dots = (float *)a.get(SCR_DOTS, (size_t)n_old * bp_max * 4);
    unsigned long long *cand = (unsigned long long *)a.get(SCR_CAND, (size_t)words * 8);
    akashic_status_t rc = (qp && dots && cand) ? AKASHIC_OK : AKASHIC_ENOMEM;
    cudaError_t e = cudaSuccess;
    for (int64_t off = 0; rc == AKASHIC_OK && off < a.n_new; off += 256) {
        const int b = (int)(a.n_new - off < 256 ? a.n_new - off : 256);
        int bp = 32;
        while (bp < b) bp <<= 1;
        k_gather_rows<<<device_sm_count(), 256, 0, st>>>(a.emb, a.row_of, a.first + off, b, bp,
                                                          a.dim, qp);
        e = cudaGetLastError();
        if (e == cudaSuccess)
            e = launch_dots(a.emb, n_old, 1, a.dim, qp, bp, 1, dots, a.status, st, launches);
        const SelectPlan sp = select_plan(n_old, bp, a.M, device_sm_count());
        if (e == cudaSuccess)
            e = launch_select_signed(sp, dots, b, cand, a.ext_of, a.first, off, a.nbr_ids,
                                     a.nbr_cos, a.status, st, launches,
                                     NsScope{nullptr, nullptr, a.dead_row});
        if (e != cudaSuccess) rc = AKASHIC_ECUDA;
        if (launches) *launches += 1;
    }
    if (rc == AKASHIC_OK && cudaStreamSynchronize(st) != cudaSuccess) rc = AKASHIC_ECUDA;
    return rc;
}

// Fused path (a6): a per-new-chunk bound from every stride-th row of the
// store, then ONE tensor-core pass over all rows x all new chunks whose
// epilogue keeps only the keys above the bounds, then an exact selection
// of the M best among them.  The dots are never written to memory.
akashic_status_t relate_top_m(const UpdateArgs &a, cudaStream_t st, int *launches) {
    // every row of the store is scored; rows holding chunks >= first are
    // masked in the selection (rows are in page order, not ID order)
    const int64_t n = a.n_rows;
    const int sms = device_sm_count();
    const int n_ct = (int)ceil_div<int64_t>(a.n_new, 256);
    const int64_t n_pad = (int64_t)n_ct * 256;
    // every stride-th row is sampled: about 512 M rows, so the bound (the
    // M-th largest sampled value) lets through about M * stride rows per
    // new chunk, which the merge stages in shared memory
    int64_t stride = n / ((int64_t)512 * a.M);
    stride = stride < 1 ? 1 : (stride > 64 ? 64 : stride);
    const int64_t n_sample = ceil_div<int64_t>(n, stride);
    const int64_t cap = 4 * (int64_t)a.M * stride > 8192 ? 4 * (int64_t)a.M * stride : 8192;
    // the sample bounds of G column tiles come from one dots GEMM that
    // writes the sampled keys column-major and one k-th launch (G tiles of
    // sampled keys: <= 512 MB)
    const int64_t tile_bytes = n_sample * 256 * 4;
    int64_t G = ((int64_t)512 << 20) / tile_bytes;
    G = G < 1 ? 1 : (G > n_ct ? n_ct : G);
    SelectPlan sp = select_plan(n_sample, (int)G * 256, a.M, sms, 1);
    sp.cap = 0;                      // no candidate buffers: bounds only
    sp.off_tr = sp.off_buf;
    sp.words = sp.off_tr + ceil_div<int64_t>(sp.n_sample * sp.bp, 2);
    uint16_t *qp = (uint16_t *)a.get(SCR_QP, (size_t)n_pad * a.dim * 2);
    int32_t *ext_s = (int32_t *)a.get(SCR_EXTS, (size_t)n_sample * 4);
    unsigned long long *ws = (unsigned long long *)a.get(SCR_WS, (size_t)sp.words * 8);
    unsigned long long *bound = (unsigned long long *)a.get(SCR_BOUND, (size_t)n_pad * 8);
    unsigned int *cnt = (unsigned int *)a.get(SCR_CNT, (size_t)n_pad * 4);
    unsigned long long *buf = (unsigned long long *)a.get(SCR_BUF, (size_t)a.n_new * cap * 8);
    akashic_status_t rc =
        (qp && ext_s && ws && bound && cnt && buf) ? AKASHIC_OK : AKASHIC_ENOMEM;
    cudaError_t e = cudaSuccess;
    bool overflow = false;
    if (rc == AKASHIC_OK) {
        k_gather_rows<<<sms * 2, 256, 0, st>>>(a.emb, a.row_of, a.first, (int)a.n_new, (int)n_pad,
                                               a.dim, qp);
        k_ext_sample<<<sms, 256, 0, st>>>(a.ext_of, n_sample, stride, ext_s);
        e = cudaGetLastError();
        // deleted chunks are never neighbours: their sample rows carry no key
        const int32_t *dead_s = nullptr;
        if (e == cudaSuccess && a.dead_row) {
            int32_t *ds = (int32_t *)a.get(SCR_DEAD_S, (size_t)n_sample * 4);
            if (!ds) {
                rc = AKASHIC_ENOMEM;
            } else {
                k_ext_sample<<<sms, 256, 0, st>>>(a.dead_row, n_sample, stride, ds);
                e = cudaGetLastError();
                dead_s = ds;
            }
        }
        for (int64_t g0 = 0; rc == AKASHIC_OK && e == cudaSuccess && g0 < n_ct; g0 += G) {
            const int gt = (int)(n_ct - g0 < G ? n_ct - g0 : G);
            const int64_t left = a.n_new - g0 * 256;
            const int b = (int)(left < (int64_t)gt * 256 ? left : (int64_t)gt * 256);
            uint32_t *keys_t = (uint32_t *)(ws + sp.off_tr);
            e = launch_dots_keys_t(a.emb, n_sample, stride, a.dim, qp + g0 * 256 * a.dim, gt,
                                   ext_s, a.first, dead_s, keys_t, a.status, st, launches);
            if (e == cudaSuccess)
                e = launch_sample_kth_keys(keys_t, n_sample, gt * 256, b, a.M, bound + g0 * 256,
                                           (unsigned int *)(ws + sp.off_cnt), st, launches);
        }
        if (rc == AKASHIC_OK && e == cudaSuccess) e = cudaMemsetAsync(cnt, 0, (size_t)n_pad * 4, st);
        if (rc == AKASHIC_OK && e == cudaSuccess)
            e = launch_dots_filter(a.emb, n, a.dim, qp, n_ct, a.n_new, a.ext_of, a.first, bound,
                                   cnt, buf, cap, a.status, st, launches, a.dead_row);
        // buffers that overflowed fall back to the exact batched path
        unsigned int max_cnt = 0;
        if (rc == AKASHIC_OK && e == cudaSuccess) {
            unsigned int *h = (unsigned int *)malloc((size_t)a.n_new * 4);
            if (!h) {
                rc = AKASHIC_ENOMEM;
            } else {
                e = cudaMemcpyAsync(h, cnt, (size_t)a.n_new * 4, cudaMemcpyDeviceToHost, st);
                if (e == cudaSuccess) e = cudaStreamSynchronize(st);
                for (int64_t c = 0; e == cudaSuccess && c < a.n_new; ++c)
                    max_cnt = h[c] > max_cnt ? h[c] : max_cnt;
                free(h);
            }
        }
        overflow = (int64_t)max_cnt > cap;
        if (e == cudaSuccess && rc == AKASHIC_OK && !overflow)
            e = launch_buf_merge_signed(cnt, buf, cap, a.n_new, a.M, a.nbr_ids, a.nbr_cos,
                                        a.status, st, launches);
        if (e == cudaSuccess && rc == AKASHIC_OK) e = cudaStreamSynchronize(st);
        if (e != cudaSuccess && rc == AKASHIC_OK) rc = AKASHIC_ECUDA;
    }
    if (rc == AKASHIC_OK && overflow) rc = relate_top_m_batched(a, st, launches);
    return rc;
}

// ------------------------------------------------------------------ CSR insert
// new degree of every row: old degree, + M for new rows, + reciprocal count
__global__ void k_new_degree(const int64_t *__restrict__ rp, int64_t n_rows, int64_t first,
                             int64_t n_new, int M, const int64_t *__restrict__ recip,
                             int64_t *__restrict__ deg) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n_rows;
         i += (int64_t)gridDim.x * blockDim.x) {
        int64_t d = rp[i + 1] - rp[i];
        if (i >= first && i < first + n_new) d += M;
        if (recip) d += recip[i];
        deg[i] = d;
    }
}

__global__ void k_count_recip(const int32_t *__restrict__ nbr, int64_t pairs,
                              unsigned long long *__restrict__ recip) {
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < pairs;
         p += (int64_t)gridDim.x * blockDim.x)
        atomicAdd(&recip[nbr[p]], 1ull);
}

// Old edges keep their order at the front of each row.  Edge-parallel:
// chunks of CHUNK_E old edges are dealt round-robin to the warps; a warp
// finds the rows of a chunk at once (chunk_rows), then issues all of a
// lane's loads for the chunk before any store; edge e of row r goes to
// nrp[r] + (e - rp[r]).
__global__ __launch_bounds__(256) void k_copy_old_rows(
    const int64_t *__restrict__ rp, const int32_t *__restrict__ col,
    const float *__restrict__ aff, int64_t n_rows, const int64_t *__restrict__ nrp,
    int32_t *__restrict__ ncol, float *__restrict__ naff, int64_t new_lo, int64_t new_hi,
    int *status) {
    __shared__ int rid_s[8][CHUNK_E];
    constexpr int PER = CHUNK_E / 32;
    const int lane = threadIdx.x & 31;
    int *rid = rid_s[threadIdx.x >> 5];
    const int64_t nnz = rp[n_rows];
    const int64_t w0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t n_chunks = (nnz + CHUNK_E - 1) / CHUNK_E;
    // chunks dealt round-robin to the warps; the lanes find the first rows
    // of a warp's next 32 chunks at once, one binary search each
    int64_t first = 0;
    int i = 0;
    for (int64_t c = w0; c < n_chunks; c += nw, ++i) {
        if ((i & 31) == 0) {
            const int64_t cl = c + (int64_t)lane * nw;
            first = cl < n_chunks ? edge_row(rp, n_rows, cl * CHUNK_E) : 0;
        }
        const int64_t base = c * CHUNK_E;
        const int64_t r_lo = __shfl_sync(0xffffffffu, first, i & 31);
        {
            int rows[PER];
            chunk_rows(rp, n_rows, nnz, base, r_lo, rid, rows);
            int32_t cv[PER];
            float av[PER];
            int64_t pos[PER];
#pragma unroll
            for (int j = 0; j < PER; ++j) {
                const int64_t e = base + 32 * j + lane;
                const int64_t row = r_lo + rows[j];
                const bool ok = e < nnz;
                cv[j] = ok ? col[e] : 0;
                av[j] = ok ? aff[e] : 0.f;
                pos[j] = ok ? e + (nrp[row] - rp[row]) : -1;
            }
#pragma unroll
            for (int j = 0; j < PER; ++j) {
                if (pos[j] < 0) continue;
                // an existing edge into a new chunk would make a reciprocal
                // edge a repeat
                if (cv[j] >= new_lo && cv[j] < new_hi) set_status(status, AKASHIC_EDEVICE);
                ncol[pos[j]] = cv[j];
                naff[pos[j]] = av[j];
            }
            __syncwarp();
        }
    }
}

// Rows of the new chunks: their M neighbours in ascending ID order (one warp
// per new row; rank of each neighbour among the row's M by ID).
__global__ void k_fill_new_rows(const int32_t *__restrict__ nbr, const float *__restrict__ cosv,
                                int64_t first, int64_t n_new, int M, float scale,
                                const int64_t *__restrict__ nrp, int32_t *__restrict__ ncol,
                                float *__restrict__ naff) {
    const int lane = threadIdx.x & 31;
    int64_t a = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t stride = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (; a < n_new; a += stride) {
        const int32_t *row = nbr + a * M;
        const int64_t o = nrp[first + a];
        for (int t = lane; t < M; t += 32) {
            const int32_t id = row[t];
            int rank = 0;
            for (int u = 0; u < M; ++u) rank += row[u] < id;
            ncol[o + rank] = id;
            naff[o + rank] = scale * cosv[a * M + t];
        }
    }
}

// Reciprocal edges j -> new chunk, appended after row j's old edges in
// ascending new-chunk order.  `order` lists the (new, slot) pair indices
// stably sorted by target j, so pairs of one j come in ascending new ID.
__global__ void k_fill_recip(const uint32_t *__restrict__ order, const uint32_t *__restrict__ tgt,
                             int64_t pairs, const int32_t *__restrict__ nbr,
                             const float *__restrict__ cosv, int64_t first, int M, float scale,
                             const int64_t *__restrict__ rp, const int64_t *__restrict__ recip_off,
                             const int64_t *__restrict__ nrp, int32_t *__restrict__ ncol,
                             float *__restrict__ naff) {
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < pairs;
         p += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t pair = order[p];
        const int64_t j = tgt[p];
        const int64_t rank = p - recip_off[j];
        const int64_t pos = nrp[j] + (rp[j + 1] - rp[j]) + rank;
        ncol[pos] = (int32_t)(first + pair / M);
        naff[pos] = scale * cosv[pair];
        (void)nbr;
    }
}

akashic_status_t csr_insert(const UpdateArgs &a, const int64_t *rp, const int32_t *col,
                            const float *aff, int64_t nnz, int64_t *new_rp, int32_t *new_col,
                            float *new_aff, cudaStream_t st, int *launches) {
    const int64_t n_rows = a.n_rows, pairs = a.n_new * a.M;
    const int sms = device_sm_count();
    const size_t tmp_bytes = (radix_tmp_bytes(pairs) > scan_tmp_bytes(n_rows + 1)
                                  ? radix_tmp_bytes(pairs)
                                  : scan_tmp_bytes(n_rows + 1)) + 4096;
    int64_t *deg = (int64_t *)a.get(SCR_DEG, (size_t)(n_rows + 1) * 8);
    int64_t *recip = (int64_t *)a.get(SCR_RECIP, (size_t)(n_rows + 1) * 8);
    int64_t *recip_off = (int64_t *)a.get(SCR_RECIP_OFF, (size_t)(n_rows + 1) * 8);
    uint32_t *keys = (uint32_t *)a.get(SCR_KEYS, (size_t)pairs * 4 + 16);
    uint32_t *vals = (uint32_t *)a.get(SCR_VALS, (size_t)pairs * 4 + 16);
    uint32_t *keys2 = (uint32_t *)a.get(SCR_KEYS2, (size_t)pairs * 4 + 16);
    uint32_t *vals2 = (uint32_t *)a.get(SCR_VALS2, (size_t)pairs * 4 + 16);
    void *tmp = a.get(SCR_TMP, tmp_bytes);
    akashic_status_t rc = (deg && recip && recip_off && keys && vals && keys2 && vals2 && tmp)
                              ? AKASHIC_OK : AKASHIC_ENOMEM;
    cudaError_t e = cudaSuccess;
    int L = 0;
    if (rc == AKASHIC_OK) {
        cudaMemsetAsync(recip, 0, (size_t)(n_rows + 1) * 8, st);
        if (a.reciprocal)
            k_count_recip<<<sms * 4, 256, 0, st>>>(a.nbr_ids, pairs, (unsigned long long *)recip);
        k_new_degree<<<sms * 4, 256, 0, st>>>(rp, n_rows, a.first, a.n_new, a.M,
                                              a.reciprocal ? recip : nullptr, deg);
        L += 3;
        e = cudaGetLastError();
        if (e == cudaSuccess) e = scan_exclusive(deg, new_rp, n_rows, tmp, tmp_bytes, st);
        if (e == cudaSuccess) {
            const int64_t warps = ceil_div<int64_t>(nnz, CHUNK_E);
            const int64_t g = ceil_div<int64_t>(warps > 0 ? warps : 1, 8);
            k_copy_old_rows<<<(unsigned)(g < (int64_t)sms * 6 ? g : (int64_t)sms * 6), 256, 0,
                              st>>>(rp, col, aff, n_rows, new_rp, new_col, new_aff, a.first,
                                    a.first + a.n_new, a.status);
            k_fill_new_rows<<<sms * 2, 256, 0, st>>>(a.nbr_ids, a.nbr_cos, a.first, a.n_new, a.M,
                                                     a.scale, new_rp, new_col, new_aff);
            L += 2;
            e = cudaGetLastError();
        }
        if (e == cudaSuccess && a.reciprocal && pairs > 0) {
            e = scan_exclusive(recip, recip_off, n_rows, tmp, tmp_bytes, st);
            if (e == cudaSuccess) e = cudaMemcpyAsync(keys, a.nbr_ids, (size_t)pairs * 4,
                                                      cudaMemcpyDeviceToDevice, st);
            if (e == cudaSuccess) e = launch_iota(vals, pairs, st);
            bool alt = false;
            int bits = 0;
            while (bits < 32 && ((int64_t)1 << bits) <= a.first - 1) ++bits;
            if (e == cudaSuccess)
                e = radix_sort_pairs(keys, vals, keys2, vals2, pairs, bits, tmp, tmp_bytes, st, &alt);
            if (e == cudaSuccess) {
                k_fill_recip<<<sms * 2, 256, 0, st>>>(alt ? vals2 : vals, alt ? keys2 : keys, pairs,
                                                      a.nbr_ids, a.nbr_cos, a.first, a.M, a.scale, rp,
                                                      recip_off, new_rp, new_col, new_aff);
                L += 1;
                e = cudaGetLastError();
            }
        }
        if (e == cudaSuccess) e = cudaStreamSynchronize(st);
        if (e != cudaSuccess) rc = AKASHIC_ECUDA;
    }
    if (launches) *launches += L;
    return rc;
}

}  // namespace ak
