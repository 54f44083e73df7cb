// Internal declarations of the relation update (a6, a7).
#pragma once

#include "ak_common.cuh"

namespace ak {

// Scratch slots of the store's grow-only update workspace.
enum UpdateScratchSlot {
    SCR_QP = 0, SCR_EXTS, SCR_WS, SCR_BOUND, SCR_CNT, SCR_BUF,              // relate (fused)
    SCR_DOTS, SCR_CAND,                                                      // relate (batched)
    SCR_DEG, SCR_RECIP, SCR_RECIP_OFF, SCR_KEYS, SCR_VALS, SCR_KEYS2, SCR_VALS2, SCR_TMP,
    SCR_NBR_IDS, SCR_NBR_COS,                                                // update results
    SCR_IN_INC, SCR_IN_DEG, SCR_IN_OFF, SCR_IN_RSTAT,                        // transpose patch
    SCR_DEAD_S,                                                              // relate sample
    SCR_DEL_KEEP, SCR_DEL_POS, SCR_DEL_TMP,                                  // deletion
    SCR_MM_G, SCR_MM_GN, SCR_MM_CAND, SCR_MM_MOVING, SCR_MM_POS, SCR_MM_PARENT,  // memory
    SCR_MM_NS, SCR_MM_IDS, SCR_MM_ROOT, SCR_MM_NSK, SCR_MM_K2, SCR_MM_V2,          // manager
    SCR_MM_TMP,
    SCR_SPLIT0, SCR_SPLIT1, SCR_SPLIT2, SCR_SPLIT3, SCR_SPLIT4, SCR_SPLIT5,  // hub plan
    SCR_SPLIT6, SCR_SPLIT7, SCR_SPLIT8, SCR_SPLIT9, SCR_SPLIT10, SCR_SPLIT11,
    SCR_COUNT
};

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
    const int32_t *dead_row;   // [n_rows] 1 for deleted chunks (never neighbours), or NULL
    int32_t *nbr_ids;      // [n_new * M] selected prior chunks, (cos desc, id asc)
    float *nbr_cos;        // [n_new * M]
    // Grow-only scratch owned by the store: scratch(ctx, slot, bytes) returns
    // a device buffer of at least `bytes` that stays allocated across calls
    // (NULL if allocation fails), so the per-call temporaries cost no
    // cudaMalloc / cudaFree once their sizes have been seen.  A call must
    // not return before its work on these buffers has finished.
    void *(*scratch)(void *ctx, int slot, size_t bytes);
    void *scratch_ctx;
    void *get(int slot, size_t bytes) const { return scratch(scratch_ctx, slot, bytes); }
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
