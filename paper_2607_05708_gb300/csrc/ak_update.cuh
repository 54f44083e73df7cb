// Internal declarations of the relation update (a6, a7).
#pragma once

#include "ak_common.cuh"

namespace ak {

struct UpdateArgs {
    const uint16_t *emb;   // store embeddings (n_rows x dim), rows in page order
    const int32_t *ext_of; // chunk ID of each row
    const int32_t *row_of; // row of each chunk ID
    int dim;
    int64_t n_rows;        // chunks in the store
    int64_t first;         // first new chunk; prior chunks are [0, first)
    int64_t n_new;         // new chunks [first, first+n_new)
    int M;                 // neighbours per new chunk
    bool reciprocal;
    float scale;           // edge logit = scale * cos
    int *status;
    int32_t *nbr_ids;      // [n_new * M] selected prior chunks, (cos desc, id asc)
    float *nbr_cos;        // [n_new * M]
};

// a6: top-M prior neighbours of every new chunk by <e_new, e_prior>.
akashic_status_t relate_top_m(const UpdateArgs &a, cudaStream_t st, int *launches);

// a7: new out-edge CSR = old edges + M out-edges per new chunk (+ reciprocal
// edges appended to the chosen rows), columns ascending in every row.
// new_rp has n_rows+1 entries; new_col/new_aff have room for the result.
akashic_status_t csr_insert(const UpdateArgs &a, const int64_t *rp, const int32_t *col,
                            const float *aff, int64_t nnz, int64_t *new_rp, int32_t *new_col,
                            float *new_aff, cudaStream_t st, int *launches);

}  // namespace ak
