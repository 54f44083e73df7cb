// Chunk deletion (the deletions D of JointCompact, Algorithm 1; invalidated
// copies are logically tombstoned, §4.2): a deleted chunk keeps its row but
// is marked dead, gets no score, is never a candidate, and every relation
// edge into or out of it is dropped from both the out-edge CSR and the
// in-edge transpose.  Compaction is edge-parallel: per-edge keep flags, one
// exclusive scan for the new positions, a scatter, and the new row pointers
// read from the scan at the old row starts.
#include "ak_common.cuh"

namespace ak {

// dead_row[row_of[id]] = 1 for every listed ID (dead_row NULL: only check);
// IDs outside [0, n_total) set EINVAL in the status word and are skipped.
__global__ void k_mark_dead(const int64_t *__restrict__ ids, int64_t n, int64_t n_total,
                            const int32_t *__restrict__ row_of, int32_t *__restrict__ dead_row,
                            int *status, const int32_t *__restrict__ page_row,
                            int32_t *__restrict__ page_live) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t id = ids[i];
        if (id < 0 || id >= n_total) {
            set_status(status, AKASHIC_EINVAL);
            continue;
        }
        if (!dead_row) continue;
        const int64_t r = row_of[id];
        if (atomicExch(&dead_row[r], 1) == 0 && page_live) atomicSub(&page_live[page_row[r]], 1);
    }
}

// keep[e] = 1 unless the edge's target (a chunk ID for the out-CSR, mapped
// to its row; a row for the transpose) or its listed source row is dead.
// The other end is handled per row by k_drop_rows.
__global__ void k_keep_by_target(const int32_t *__restrict__ tgt, int64_t nnz,
                                 const int32_t *__restrict__ row_of,
                                 const int32_t *__restrict__ dead_row, int64_t *__restrict__ keep) {
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < nnz;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int32_t t = tgt[e];
        keep[e] = dead_row[row_of ? row_of[t] : t] ? 0 : 1;
    }
}

// Every edge of the listed IDs' own rows is dropped (their out-edges in the
// out-CSR, their in-edges in the transpose): one warp per deleted chunk.
__global__ void k_drop_rows(const int64_t *__restrict__ ids, int64_t n, int64_t n_total,
                            const int32_t *__restrict__ row_of, const int64_t *__restrict__ ptr,
                            int64_t *__restrict__ keep) {
    const int lane = threadIdx.x & 31;
    int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t stride = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (; i < n; i += stride) {
        const int64_t id = ids[i];
        if (id < 0 || id >= n_total) continue;
        const int64_t r = row_of ? row_of[id] : id;
        for (int64_t e = ptr[r] + lane; e < ptr[r + 1]; e += 32) keep[e] = 0;
    }
}

__global__ void k_compact_edges(const int64_t *__restrict__ keep, const int64_t *__restrict__ pos,
                                int64_t nnz, const int32_t *__restrict__ a_in,
                                const float *__restrict__ b_in, int32_t *__restrict__ a_out,
                                float *__restrict__ b_out) {
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < nnz;
         e += (int64_t)gridDim.x * blockDim.x) {
        if (!keep[e]) continue;
        a_out[pos[e]] = a_in[e];
        b_out[pos[e]] = b_in[e];
    }
}

__global__ void k_new_ptr(const int64_t *__restrict__ ptr, const int64_t *__restrict__ pos,
                          int64_t n, int64_t *__restrict__ new_ptr) {
    for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r <= n;
         r += (int64_t)gridDim.x * blockDim.x)
        new_ptr[r] = pos[ptr[r]];
}

// Edges handed to an append may not point at a deleted chunk (targets below
// `first`; the batch's own chunks cannot be deleted yet).
__global__ void k_check_dead_targets(const int32_t *__restrict__ col, int64_t nnz, int64_t first,
                                     const int32_t *__restrict__ row_of,
                                     const int32_t *__restrict__ dead_row, int *status) {
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < nnz;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int32_t c = col[e];
        if (c >= 0 && (int64_t)c < first && dead_row[row_of[c]]) set_status(status, AKASHIC_EDEVICE);
    }
}

cudaError_t launch_check_dead_targets(const int32_t *col, int64_t nnz, int64_t first,
                                      const int32_t *row_of, const int32_t *dead_row, int *status,
                                      cudaStream_t st) {
    if (nnz <= 0) return cudaSuccess;
    k_check_dead_targets<<<device_sm_count() * 4, 256, 0, st>>>(col, nnz, first, row_of, dead_row,
                                                                status);
    return cudaGetLastError();
}

cudaError_t launch_mark_dead(const int64_t *ids, int64_t n, int64_t n_total, const int32_t *row_of,
                             int32_t *dead_row, int *status, cudaStream_t st,
                             const int32_t *page_row, int32_t *page_live) {
    if (n <= 0) return cudaSuccess;
    k_mark_dead<<<device_sm_count(), 256, 0, st>>>(ids, n, n_total, row_of, dead_row, status,
                                                   page_row, page_live);
    return cudaGetLastError();
}

cudaError_t launch_drop_dead_edges(const DropDead &d, cudaStream_t st) {
    const int sms = device_sm_count();
    if (d.nnz > 0) {
        k_keep_by_target<<<sms * 8, 256, 0, st>>>(d.tgt, d.nnz, d.tgt_row_of, d.dead_row, d.keep);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        if (d.n_ids > 0) {
            k_drop_rows<<<sms * 2, 256, 0, st>>>(d.ids, d.n_ids, d.n_total, d.own_row_of, d.ptr,
                                                 d.keep);
            e = cudaGetLastError();
            if (e != cudaSuccess) return e;
        }
    }
    // keep[nnz] = 0 so that pos[nnz] is the surviving count
    cudaError_t e = cudaMemsetAsync(d.keep + d.nnz, 0, 8, st);
    if (e == cudaSuccess) e = scan_exclusive(d.keep, d.pos, d.nnz + 1, d.tmp, d.tmp_bytes, st);
    if (e != cudaSuccess) return e;
    if (d.nnz > 0) {
        k_compact_edges<<<sms * 8, 256, 0, st>>>(d.keep, d.pos, d.nnz, d.tgt, d.val, d.tgt_out,
                                                 d.val_out);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    k_new_ptr<<<sms * 4, 256, 0, st>>>(d.ptr, d.pos, d.n_rows, d.ptr_out);
    return cudaGetLastError();
}

}  // namespace ak
