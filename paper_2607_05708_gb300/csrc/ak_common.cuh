// Internal declarations shared by the library's translation units.
// Nothing here is part of the public ABI (include/akashic_mem.h is).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/akashic_mem.h"

namespace ak {

// ------------------------------------------------------------------ status word
// Device-side faults are recorded with atomicCAS(status, 0, code) so that the
// first one wins; the host reads and clears the word in akashic_mem_sync.
__device__ __forceinline__ void set_status(int *status, int code) {
    if (status) atomicCAS(status, 0, code);
}

// ------------------------------------------------------------------ dependent launches
// The retrieval's kernels are launched with programmatic stream
// serialisation (launch_pdl): each may be scheduled while the kernel before
// it in the stream drains, and waits here, before it touches global memory,
// until that kernel has completed and its writes are visible (a kernel
// launched without the attribute returns from the wait at once).
__device__ __forceinline__ void griddep_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// ------------------------------------------------------------------ small helpers
__device__ __forceinline__ float bf16_to_f32(uint16_t h) {
    return __uint_as_float(((uint32_t)h) << 16);
}

template <typename T>
__host__ __device__ __forceinline__ T ceil_div(T a, T b) { return (a + b - 1) / b; }

// Selection key: larger key = better.  High word: the score's fp32 bit
// pattern (scores are >= 0, where the bit pattern is monotone in value);
// low word: ~id, so that on equal scores the lower chunk ID wins.
__device__ __forceinline__ unsigned long long make_key(float score, uint32_t id) {
    return ((unsigned long long)__float_as_uint(score) << 32) | (unsigned long long)(~id);
}
__device__ __forceinline__ float key_score(unsigned long long key) {
    return __uint_as_float((uint32_t)(key >> 32));
}
__device__ __forceinline__ uint32_t key_id(unsigned long long key) {
    return ~(uint32_t)(key & 0xffffffffull);
}

// Candidate scope of a selection.  Namespaces (§4.1: the candidates of a
// query are the chunks of the caller's (user_id, session_id) table): row j
// is a candidate for query column c only if ns_row[j] == q_ns[c]
// (q_ns == NULL: no namespace scope).  Deletions (tombstones): a row with
// dead[j] != 0 is never a candidate (dead == NULL: none deleted).
struct NsScope {
    const int32_t *ns_row;   // [rows] tag of the chunk in each row (or sample row)
    const int32_t *q_ns;     // [bp] tag of each query column
    const int32_t *dead;     // [rows] 1 where the chunk was deleted
};
__device__ __forceinline__ bool in_scope(const NsScope &s, int64_t row, int col) {
    return (!s.dead || !s.dead[row]) && (!s.q_ns || s.ns_row[row] == s.q_ns[col]);
}
__host__ __device__ __forceinline__ bool scope_active(const NsScope &s) {
    return s.q_ns != nullptr || s.dead != nullptr;
}

// Split-bf16 of two fp32 values: hi = bf16(x) (round to nearest), lo =
// bf16(x - hi) (x - hi is exact in fp32), packed two to a word (x in the low
// half); x = hi + lo to within 2^-17 relative.
__device__ __forceinline__ uint32_t split_bf16_pair(float x, float y, uint32_t &lo) {
    const __nv_bfloat16 hx = __float2bfloat16_rn(x), hy = __float2bfloat16_rn(y);
    const __nv_bfloat16 lx = __float2bfloat16_rn(x - __bfloat162float(hx));   // exact rest
    const __nv_bfloat16 ly = __float2bfloat16_rn(y - __bfloat162float(hy));
    lo = (uint32_t)__bfloat16_as_ushort(lx) | ((uint32_t)__bfloat16_as_ushort(ly) << 16);
    return (uint32_t)__bfloat16_as_ushort(hx) | ((uint32_t)__bfloat16_as_ushort(hy) << 16);
}

// log2(e): scores exp(tau x - c) are evaluated as 2^(x tau log2(e) - c log2(e))
// (one FMA and the hardware exp2).
constexpr float LOG2E_F = 1.44269504088896340736f;

// Keys for signed cosine values: order-preserving map of any finite fp32 to
// uint32 (flip all bits of negatives, set the sign bit of non-negatives).
__device__ __forceinline__ uint32_t ordered_bits(float v) {
    uint32_t u = __float_as_uint(v);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float unordered_bits(uint32_t o) {
    uint32_t u = (o & 0x80000000u) ? (o & 0x7fffffffu) : ~o;
    return __uint_as_float(u);
}

// Set the thread-local message returned by akashic_mem_last_error().
void set_last_error(const char *msg);

// ------------------------------------------------------------------ launchers
// All launchers enqueue on `st` and report launch errors by return value.

// Score (a1) on the tensor cores: u[j, c] = exp(tau * <e_j, q_c> - shift[c])
// for j < n, c < bp (bp = 32, 64, 128 or 256), written chunk-major with row
// stride bp; zpart[r, c] = sum of u over the rows handled by score CTA r,
// for r < *zrows.  score_tiles(n) bounds *zrows.
int64_t score_tiles(int64_t n);
// dead_row (or NULL): rows of deleted chunks score u = 0 (no part in Z).
// row_max / row_min (optional, together): [n] the largest and smallest u of
// each row over the first n_real columns (the real queries), for the
// propagation's row bounds; with them, ext (optional, [2], zeroed before)
// gets their extremes in launch_final_bounds' encoding.
// One thread waits on a barrier that nothing signals, giving up after
// `polls` polls like every bounded wait (ETIMEOUT into *status).
cudaError_t launch_wait_timeout_check(int *status, uint32_t polls, cudaStream_t st);
// Raises the score kernel's shared-memory limit for every query width on the
// current device now (launch_score does it lazily per width otherwise).
cudaError_t prepare_score_gemm();
cudaError_t launch_score(const uint16_t *emb, int64_t n, int dim, const uint16_t *qp, int bp,
                         const float *shift, float tau, float *u, float *zpart, int *status,
                         cudaStream_t st, int *launches, int *zrows,
                         const int32_t *dead_row = nullptr, float *row_max = nullptr,
                         float *row_min = nullptr, int n_real = 0, unsigned int *ext = nullptr);
// The same scores with u written as split bf16 instead of fp32: u_hi and u_lo
// [n][bp] each, u = hi + lo to within 2^-17 relative (the operand form the
// candidates' tensor-core pass reads); Z's column sums from the fp32 values.
cudaError_t launch_score_split(const uint16_t *emb, int64_t n, int dim, const uint16_t *qp, int bp,
                               const float *shift, float tau, uint16_t *u_hi, uint16_t *u_lo,
                               float *zpart, int *status, cudaStream_t st, int *launches,
                               int *zrows, const int32_t *dead_row, float *row_max,
                               float *row_min, int n_real, unsigned int *ext);

// The score on every stride-th row only: out[v, c] = u[v*stride, c] for
// v < n_sample (same kernel and arithmetic as launch_score, so the values
// are those the full pass computes); zpart receives partial sums of the
// sample (scratch, one row per CTA, at most score_tiles(n_sample) rows).
cudaError_t launch_score_sample(const uint16_t *emb, int64_t n_sample, int64_t stride, int dim,
                                const uint16_t *qp, int bp, const float *shift, float tau,
                                float *out, float *zpart, int *status, cudaStream_t st,
                                int *launches);
// Score with the top-k filter fused and no slab written: zpart as in
// launch_score; the key (u bits, chunk ID ext_of[j]) of every (j, c) with
// c < n_cols that is >= bound[c] is appended to buf[c][...] (count cnt[c],
// capacity cap).
cudaError_t launch_score_filter(const uint16_t *emb, int64_t n, int dim, const uint16_t *qp,
                                int bp, int64_t n_cols, const float *shift, float tau,
                                float *zpart, const int32_t *ext_of,
                                const unsigned long long *bound, unsigned int *cnt,
                                unsigned long long *buf, int64_t cap, NsScope ns, int *status,
                                cudaStream_t st, int *launches, int *zrows);

// Plain dot products out[j, c] = <e_{j*row_stride}, q_c> (bf16 tensor
// cores, fp32 accumulate) for j < n and the n_ctiles * bp columns of qp;
// row stride n_ctiles * bp in out.
cudaError_t launch_dots(const uint16_t *emb, int64_t n, int64_t row_stride_rows, int dim,
                        const uint16_t *qp, int bp, int n_ctiles, float *out, int *status,
                        cudaStream_t st, int *launches);
// Fused relation top-M filter: dots of every row j < n against the
// n_ctiles*256 rows of qp; the selection key (signed dot, chunk ID
// ext_of[j]) of every (j, c) with c < n_cols and ext_of[j] < id_limit that
// is >= bound[c] is appended to buf[c][...] (count cnt[c], capacity cap).
cudaError_t launch_dots_filter(const uint16_t *emb, int64_t n, int dim, const uint16_t *qp,
                               int n_ctiles, int64_t n_cols, const int32_t *ext_of,
                               int64_t id_limit, const unsigned long long *bound,
                               unsigned int *cnt, unsigned long long *buf, int64_t cap,
                               int *status, cudaStream_t st, int *launches,
                               const int32_t *dead_row = nullptr);

// Sampled dots as selection keys, column-major: keys_t[c][j] for the rows
// j < n (row j*row_stride of emb) and the n_ctiles*256 rows c of qp; the
// key is the order-preserving bits of the signed dot, or 0 where row j is
// deleted (dead_row[j], if given) or ext_of[j] >= id_limit.
cudaError_t launch_dots_keys_t(const uint16_t *emb, int64_t n, int64_t row_stride_rows, int dim,
                               const uint16_t *qp, int n_ctiles, const int32_t *ext_of,
                               int64_t id_limit, const int32_t *dead_row, uint32_t *keys_t,
                               int *status, cudaStream_t st, int *launches);

// Query preparation: pad q (b rows) to bp rows of zeros and compute
// shift[c] = tau * |q_c| * max_norm (0 for padding); flags ERANGE.
// ext_zero (or NULL): two words set to 0 (the row extremes' initial value).
cudaError_t launch_prep_queries(const uint16_t *q, int b, int bp, int dim, float tau,
                                const float *max_norm, uint16_t *qp, float *shift, int *status,
                                cudaStream_t st, unsigned int *ext_zero = nullptr);

// Running maximum of row norms of emb[0..n) into *max_norm (monotone).
cudaError_t launch_row_norm_max(const uint16_t *emb, int64_t n, int dim, float *max_norm,
                                cudaStream_t st);

// ------------------------------------------------------------------ graph
int device_sm_count();

// Propagation work plan.  Rows with more than SPLIT_T in-edges (the hubs of
// a power-law relation graph) are cut into segments of at most SEG_LEN
// edges that never cross a source window of WIN_ROWS rows; segments are
// processed window by window so that the source rows they gather stay in L2,
// and a fixup pass sums each hub's segment partials in order.
struct SplitParams {
    int64_t split_t = 256;      // in-degree above which a row is split
    int64_t seg_len = 512;      // edges per segment at most
    int64_t win_rows = 32768;   // source window (rows); 32 MB of slab at 256 queries
};
constexpr int ROWS_PER_GRAB = 8;     // rows a warp claims at a time (dynamic scheduling)

// Exclusive prefix sum of `in` (n values) into out (n+1 values; out[n] = total).
// `launches`, if given, is incremented by the kernels launched.
cudaError_t scan_exclusive(const int64_t *in, int64_t *out, int64_t n, void *tmp,
                           size_t tmp_bytes, cudaStream_t st, int *launches = nullptr);
size_t scan_tmp_bytes(int64_t n);

// Stable LSD radix sort of (key, value) pairs on the low `bits` key bits;
// the result lands in (keys, vals) or, if *result_in_alt, in the alt buffers.
size_t radix_tmp_bytes(int64_t n);
cudaError_t radix_sort_pairs(uint32_t *keys, uint32_t *vals, uint32_t *keys_alt,
                             uint32_t *vals_alt, int64_t n, int bits, void *tmp,
                             size_t tmp_bytes, cudaStream_t st, bool *result_in_alt,
                             int *launches = nullptr);

// CSR helpers (see ak_graph.cu).
cudaError_t launch_edge_src_check(const int64_t *row_ptr, const int32_t *col, int64_t n_rows,
                                  int64_t row_base, int64_t n_total, int32_t *src, int *status,
                                  cudaStream_t st);
// w = row softmax of the logits, per row: w_e = exp(aff_e - max) * inv with
// inv = 1 / sum exp(aff - max); (max, inv) of row r go to rstat[r] when
// rstat is not NULL, so that any copy of a weight (the in-edge transpose)
// can be recomputed bit for bit by row_softmax_weight.
__device__ __forceinline__ float row_softmax_weight(float aff, float2 stat) {
    return expf(aff - stat.x) * stat.y;
}
cudaError_t launch_row_softmax(const int64_t *row_ptr, const float *aff, float *w, int64_t n_rows,
                               float2 *rstat, cudaStream_t st);
// Edge-parallel moves of CSR rows: a warp takes CHUNK_E consecutive edges
// [base, base + CHUNK_E), lane l the edges base + 32 j + l (j < CHUNK_E / 32),
// and finds their rows without a search per edge.  Given r_lo, the row of
// edge `base` (ptr[r_lo] <= base < ptr[r_lo + 1]), the warp marks in its own
// shared array rid[] the first edge of every later row that starts inside
// the chunk, as row - r_lo (where several rows start at one edge, the empty
// rows before it, the largest wins); a running maximum over the positions,
// taken 32 at a time across the lanes, gives every edge its row:
// rows[j] = row of edge base + 32 j + lane - r_lo.  ptr has n + 1 entries,
// ptr[n] = nnz.
// All 32 lanes call it.  Chunks are small (four edges a lane) so that the
// moving kernels stay at high occupancy: their loads are latency-bound.
constexpr int CHUNK_E = 128;
__device__ __forceinline__ void chunk_rows(const int64_t *__restrict__ ptr, int64_t n,
                                           int64_t nnz, int64_t base, int64_t r_lo, int *rid,
                                           int (&rows)[CHUNK_E / 32]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int j = 0; j < CHUNK_E / 32; ++j) rid[32 * j + lane] = 0;
    __syncwarp();
    // rows starting at or past nnz own no edge (the empty rows at the end)
    const int64_t lim = base + CHUNK_E < nnz ? base + CHUNK_E : nnz;
    for (int64_t r0 = r_lo + 1; r0 < n; r0 += 32) {
        const int64_t r = r0 + lane;
        const int64_t s = r < n ? ptr[r] : INT64_MAX;   // > base for every r > r_lo
        if (s < lim) atomicMax(&rid[s - base], (int)(r - r_lo));
        if (__shfl_sync(0xffffffffu, s, 31) >= lim) break;
    }
    __syncwarp();
    int carry = 0;
#pragma unroll
    for (int j = 0; j < CHUNK_E / 32; ++j) {
        int x = max(rid[32 * j + lane], carry);
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x = max(x, t);
        }
        rows[j] = x;
        carry = __shfl_sync(0xffffffffu, x, 31);
    }
    __syncwarp();
}
// The row of edge e (e < ptr[n]) by binary search: the largest r with
// ptr[r] <= e.
__device__ __forceinline__ int64_t edge_row(const int64_t *__restrict__ ptr, int64_t n,
                                            int64_t e) {
    int64_t lo = 0, hi = n;
    while (hi - lo > 1) {
        const int64_t mid = (lo + hi) >> 1;
        if (ptr[mid] <= e) lo = mid;
        else hi = mid;
    }
    return lo;
}
// The store keeps chunks in HBM in page order: row r holds chunk ext_of[r],
// chunk c lives in row row_of[c].  The out-edge CSR stays in chunk IDs; the
// in-edge transpose used by propagation is in rows.
cudaError_t launch_in_degree(const int32_t *col, const int32_t *row_of, int64_t nnz, int64_t *deg,
                             cudaStream_t st);
cudaError_t launch_iota(uint32_t *v, int64_t n, cudaStream_t st);
// out[row_of[first + i]] = in[i], i < n.
cudaError_t launch_scatter_by_row(const int32_t *in, const int32_t *row_of, int64_t first,
                                  int64_t n, int32_t *out, cudaStream_t st);
cudaError_t launch_map_keys(const uint32_t *sel, const int32_t *ids, const int32_t *row_of,
                            uint32_t *keys, int64_t n, cudaStream_t st);
cudaError_t launch_gather_in(const uint32_t *order, const int32_t *src, const int32_t *row_of,
                             const float *w, const float *aff, int32_t *in_src, float *in_w,
                             float *in_aff, int64_t nnz, cudaStream_t st);

// Incremental in-edge transpose after a relation update (ak_inedges.cu).
struct InEdgeUpdate {
    int64_t n;                          // store rows (new chunks included)
    int64_t nnz_new;                    // edges after the update
    const int64_t *in_ptr_old;          // [n+1]
    const int32_t *in_src_old;
    const float *in_aff_old;
    int64_t *in_ptr_new;                // [n+1]
    int32_t *in_src_new;                // [nnz_new]
    float *in_aff_new, *in_w_new;       // [nnz_new]
    const int32_t *nbr_ids;             // [n_new][M] chosen prior chunk IDs
    const float *nbr_cos;               // [n_new][M]
    float scale;                        // logit = scale * cos
    int64_t first, n_new;
    int M;
    bool reciprocal;
    int row_bits;                       // key bits of a row index
    const int32_t *row_of, *ext_of;
    const float2 *rstat;                // per chunk ID: (max, inv) of its out-row
};
// The update writes in_w_new for every edge as it places it (old edges
// moved, new edges placed): row_softmax_weight(aff, rstat[ext_of[src]]).
struct InEdgeScratch {
    int64_t *inc, *deg, *fwd_off;       // [n+1] each
    uint32_t *keys, *vals, *keys2, *vals2;   // [n_new * M] each
    void *tmp;
    size_t tmp_bytes;                   // >= radix and scan needs
    float2 *rstat_row;                  // [n]: rstat[ext_of[r]], the statistics by row
};
cudaError_t launch_in_edges_update(const InEdgeUpdate &u, const InEdgeScratch &s, cudaStream_t st,
                                   int *launches);
// in_w[e] = row_softmax_weight(in_aff[e], rstat[ext_of[in_src[e]]])
cudaError_t launch_in_weights(const int32_t *in_src, const float *in_aff, int64_t nnz,
                              const int32_t *ext_of, const float2 *rstat, float *in_w,
                              cudaStream_t st);
cudaError_t launch_batch_layout(const uint32_t *order, int64_t first, int64_t n, int dim,
                                const uint16_t *emb_in, uint16_t *emb, const int32_t *page_in,
                                int64_t first_page, int per_page, int32_t *page_row,
                                int32_t *ext_of, int32_t *row_of, cudaStream_t st);
// Split plan (see SPLIT_T): per row the number of segments (0 for rows kept
// whole) and a split flag; then the segments themselves with their window.
cudaError_t launch_split_count(const SplitParams &sp, const int64_t *in_ptr, const int32_t *in_src,
                               int64_t n, int64_t *nseg, int64_t *flag, cudaStream_t st);
cudaError_t launch_split_fill(const SplitParams &sp, const int64_t *in_ptr, const int32_t *in_src,
                              int64_t n,
                              const int64_t *nseg, const int64_t *slot_off,
                              const int64_t *split_idx, int32_t *split_row, int64_t *split_slot0,
                              int64_t *seg_e0, int64_t *seg_e1, uint32_t *seg_win,
                              cudaStream_t st);
// Permute segments into window-major order: dst[i] = src[order[i]], slot[i] = order[i].
cudaError_t launch_seg_permute(const uint32_t *order, const int64_t *e0, const int64_t *e1,
                               int64_t n_segs, int64_t *e0s, int64_t *e1s, int32_t *slot,
                               cudaStream_t st);

// keys[r] = ~(slot count of split row r), vals[r] = r (sorted: heaviest first).
cudaError_t launch_split_keys(const int64_t *slot0, int64_t n_split, uint32_t *keys,
                              uint32_t *vals, cudaStream_t st);

// Memory Manager tables (ak_mm.cu): the page directory's slot counters,
// the co-retrieval statistics and the running counters.
struct MmTables {
    int32_t *page_total, *page_live;   // [page capacity] slots used / live chunks per page
    int32_t *sel;                      // [chunk capacity] requests that retrieved the chunk
    unsigned long long *co_key;        // [co_cap] chunk pair (lo << 32 | hi), ~0 = empty
    uint32_t *co_val;                  // [co_cap] requests that retrieved both
    int64_t co_cap;                    // power of two
    int64_t *next_page;                // device copy of the next fresh page ID
    int64_t *writes;                   // chunks written (appends, relocations, compaction)
    unsigned long long *released;      // pages released by the last compaction
};
cudaError_t launch_mm_count(const int64_t *S, int n_req, int s_len, int64_t n,
                            const int32_t *row_of, const int32_t *dead_row, const MmTables &t,
                            int *status, cudaStream_t st);
// g_buf [n_req][64], g_n [n_req] scratch.
cudaError_t launch_mm_relocate(const int64_t *S, int n_req, int s_len, int64_t n,
                               const int32_t *row_of, const int32_t *dead_row, int32_t *page_row,
                               const MmTables &t, float tau, int per_page, int32_t *g_buf,
                               int32_t *g_n, cudaStream_t st);
cudaError_t launch_mm_compact_prepare(const MmTables &t, int64_t n_pages, float theta, int64_t n,
                                      const int32_t *row_of, const int32_t *dead_row,
                                      const int32_t *page_row, int32_t *cand, int64_t *moving,
                                      int32_t *parent, cudaStream_t st);
cudaError_t launch_mm_union(const MmTables &t, const int64_t *moving, const int32_t *ns_by_id,
                            float tau, int32_t *parent, int *status, cudaStream_t st);
cudaError_t launch_mm_keys(const int64_t *moving, const int64_t *pos, int64_t n,
                           const int32_t *parent, const int32_t *ns_by_id, uint32_t *ids,
                           uint32_t *root_key, uint32_t *ns_key, cudaStream_t st);
// part_pages[i] = pages the namespace run starting at i fills (0 inside a run)
cudaError_t launch_mm_part_pages(const uint32_t *ns_sorted, int64_t count, int per_page,
                                 int64_t *part_pages, cudaStream_t st);
// releases the candidate pages, then writes the ordered chunks into fresh
// pages from first_page on, each namespace from its own base page
cudaError_t launch_mm_release_repack(const MmTables &t, int64_t n_pages, const int32_t *cand,
                                     const uint32_t *order_ids, const uint32_t *ns_sorted,
                                     const int64_t *part_base, int64_t count,
                                     const int32_t *row_of, int32_t *page_row, int64_t first_page,
                                     int per_page, cudaStream_t st);
cudaError_t launch_mm_count_pages(const int32_t *page_row, int64_t first, int64_t n,
                                  const MmTables &t, cudaStream_t st);
// out[0..2] = pages in use, slots in use, live slots
cudaError_t launch_mm_stats(const MmTables &t, int64_t n_pages, unsigned long long *out,
                            cudaStream_t st);
cudaError_t launch_mm_rehash(const unsigned long long *old_key, const uint32_t *old_val,
                             int64_t old_cap, const MmTables &t, int *status, cudaStream_t st);
// out[i] = ns_by_id[ids[i]] as an order-preserving unsigned key
cudaError_t launch_mm_ns_keys(const uint32_t *ids, int64_t count, const int32_t *ns_by_id,
                              uint32_t *out, cudaStream_t st);
// out[c] = by_row[row_of[c]], c < n
cudaError_t launch_by_id(const int32_t *by_row, const int32_t *row_of, int64_t n, int32_t *out,
                         cudaStream_t st);

// Chunk deletion (ak_delete.cu).  dead_row[row_of[id]] = 1 for the listed
// IDs (out-of-range IDs set EINVAL in *status and are skipped; dead_row
// NULL: check only).
// A newly deleted chunk's slot becomes invalid: page_live[page_row[row]]
// drops by one (page_row / page_live may be NULL).
cudaError_t launch_mark_dead(const int64_t *ids, int64_t n, int64_t n_total, const int32_t *row_of,
                             int32_t *dead_row, int *status, cudaStream_t st,
                             const int32_t *page_row = nullptr, int32_t *page_live = nullptr);
// EDEVICE in *status if any col[e] < first names a deleted chunk.
cudaError_t launch_check_dead_targets(const int32_t *col, int64_t nnz, int64_t first,
                                      const int32_t *row_of, const int32_t *dead_row, int *status,
                                      cudaStream_t st);
// One CSR without the edges that touch a dead row: an edge survives if its
// target (tgt[e], mapped through tgt_row_of unless NULL) is not dead and it
// is not in the row of a listed ID (rows found through own_row_of unless
// NULL).  Survivors keep their order; ptr_out[r] = new start of row r.
struct DropDead {
    int64_t n_rows, nnz;
    const int64_t *ptr;                 // [n_rows+1]
    const int32_t *tgt;                 // [nnz]
    const float *val;                   // [nnz] carried along (logits)
    const int32_t *tgt_row_of;          // chunk ID -> row for targets, or NULL (targets are rows)
    const int32_t *dead_row;            // [rows]
    const int64_t *ids;                 // [n_ids] deleted chunk IDs
    int64_t n_ids, n_total;
    const int32_t *own_row_of;          // chunk ID -> row of the CSR, or NULL (CSR rows are IDs)
    int64_t *keep, *pos;                // scratch [nnz+1] each
    void *tmp;                          // scan scratch
    size_t tmp_bytes;
    int64_t *ptr_out;                   // [n_rows+1]
    int32_t *tgt_out;                   // [nnz]
    float *val_out;                     // [nnz]
};
cudaError_t launch_drop_dead_edges(const DropDead &d, cudaStream_t st);

// Propagation hop (a2): out[j,:] = u[j,:] + alpha * sum_{i->j} w_ij * in[i,:].
struct HopPlan {
    SplitParams split;
    const int64_t *in_ptr;      // n+1
    const int32_t *in_src;      // nnz
    const float *in_w;          // nnz
    int64_t n;
    // rows whose in-degree exceeds the segment length are split
    int64_t n_split_rows;       // number of such rows
    const int32_t *split_row;   // [n_split_rows] row index
    const int64_t *split_slot0; // [n_split_rows+1] first partial slot of each split row
    int64_t n_segs;             // total segments of split rows (= partial slots)
    const int64_t *seg_e0;      // [n_segs] first edge, window-major order
    const int64_t *seg_e1;      // [n_segs] end edge
    const int32_t *seg_slot;    // [n_segs] partial slot (segments of a row are contiguous)
    const int32_t *split_order; // [n_split_rows] split rows by slot count, largest first
    const int32_t *slot_split;  // [n_segs] split row owning each partial slot
};
// Top-k filter fused into a hop's output: every written value whose key
// (score bits, ~chunk ID) is >= bound[column] is appended to that column's
// buffer, as the selection's filter pass would (see ak_select.cu).
struct HopFilter {
    const int32_t *ext_of;            // row -> chunk ID
    const unsigned long long *bound;  // [bp]
    unsigned int *cnt;                // [bp]
    unsigned long long *buf;          // [bp][cap]
    int64_t cap;
    NsScope ns;                       // candidates only within the query's namespace
};
// Row bounds for the last hop, whose output only feeds the fused top-k
// filter: row_ub[j] bounds every real query column's fp32 value of the
// hop's output s_j from above (launch_row_bounds), `floor` is at most every
// real query's k-th largest final value (launch_prune_floor); a row with
// row_ub < floor appends nothing in any column and is skipped, so the
// filter's output is unchanged.
struct HopBound {
    const float *row_ub;       // [n]
    const float *floor;        // device scalar
    const int32_t *split_skip; // [n_split_rows] split rows to skip (launch_split_flags)
    const int32_t *slot_skip;  // [n_segs] their partial slots
    const int32_t *kept_rows;  // [n] rows kept whole that reach the floor ...
    const int64_t *kept_count; // ... [0] their number, [1] that of kept_segs (device)
    const int32_t *kept_segs;  // [n_segs] segments of the unpruned split rows
};
// Scratch of the kept lists' compaction: flag / pos [max(n, n_segs) + 1]
// int64, tmp of scan_tmp_bytes(max(n, n_segs)) bytes.
struct KeptScratch {
    int64_t *flag, *pos;
    void *tmp;
    size_t tmp_bytes;
};
// Graph-only mass vectors for the row bounds, levels t0..t1 (level 0, all
// ones, already in place): mup[t] >= g (1 + eps) sum_i w_ij mup[t-1]_i and
// mdn[t] <= g' (1 - eps) sum_i w_ij mdn[t-1]_i, g / g' the rounding growth of
// a hop's sum over the row's edges.  mup / mdn are [levels + 1][n];
// `zeros` is [n]; split_vu/vl [n_split_rows] scratch.  With them, for every
// real query column (U0 / L0 u's row maxima / minima, Umax / Lmin their
// extremes over the live rows):
//   s^(H)_j <= (U0_j + Umax sum_{t<=H} alpha^t mup[t]_j) (1 + eps),
//   s^(H)_j >= (L0_j + Lmin sum_{t<=H} alpha^t mdn[t]_j) (1 - eps)
// (by induction over the hops: every source's value lies in
// [Lmin (1 + ...), Umax (1 + ...)]).
cudaError_t launch_mass_levels(const HopPlan &p, int t0, int t1, float *mup, float *mdn,
                               const float *zeros, float *split_vu, float *split_vl,
                               cudaStream_t st);
// The row bounds of the last hop's output (one row; k_final_bounds writes
// them for every row, the reach path evaluates them where it needs them):
// ub_j = (U0_j + Umax sum_t alpha^t Mup[t]_j)(1 + 1e-5),
// lb_j = (L0_j + Lmin sum_t alpha^t Mdn[t]_j)(1 - 1e-5), Horner over t.
__device__ __forceinline__ float row_upper_bound(const float *u0, const float *mup, int64_t n,
                                                 int H, float alpha, float umax, int64_t j) {
    float c = 0.f;
    for (int t = H; t >= 1; --t) c = alpha * (c + __ldg(mup + (int64_t)t * n + j));
    return fmaf(umax, c, u0[j]) * (1.f + 1e-5f);
}
__device__ __forceinline__ float row_lower_bound(const float *l0, const float *mdn, int64_t n,
                                                 int H, float alpha, float lmin, int64_t j) {
    if (!(lmin < INFINITY)) return 0.f;
    float c = 0.f;
    for (int t = H; t >= 1; --t) c = alpha * (c + __ldg(mdn + (int64_t)t * n + j));
    return fmaf(lmin, c, l0[j]) * (1.f - 1e-5f);
}
__device__ __forceinline__ float ext_umax(const unsigned int *ext) { return __uint_as_float(ext[0]); }
__device__ __forceinline__ float ext_lmin(const unsigned int *ext) {
    return __uint_as_float(0x7f800000u - ext[1]);
}
// Per call: ub / lb [n] from u's row extremes u0 / l0 and the mass levels
// 1..H.  ext [2]: ext[0] the bits of Umax = max_j u0_j, ext[1] 0x7f800000
// minus the bits of Lmin = min over u0_j > 0 of l0_j (both maxima, so zero
// is the empty value); computed here unless ext_ready (the score GEMM's
// epilogue already reduced them).
cudaError_t launch_final_bounds(const float *u0, const float *l0, const float *mup,
                                const float *mdn, int64_t n, int H, float alpha,
                                unsigned int *ext, float *ub, float *lb, cudaStream_t st,
                                int *launches, bool ext_ready = false);
// Floors of a namespace-scoped last hop: a row can only be selected by the
// batch's queries of its own namespace, so its floor is that namespace's
// (tag_floor[i] for tags[i] == its tag; the tags are the batch's distinct
// query namespaces, ascending), or +inf when no query of the batch has its
// namespace.  ns_row == NULL: the one device floor applies to every row.
struct NsFloors {
    const int32_t *ns_row;    // [n] namespace tag of each row
    const int32_t *tags;      // [<= PF_TAGS] distinct query tags, ascending
    const int *n_tags;        // their number (device)
    const float *tag_floor;   // [<= PF_TAGS]
};
constexpr int PF_TAGS = 256;
__device__ __forceinline__ float row_floor(const NsFloors &f, float floor_, int64_t row) {
    if (!f.ns_row) return floor_;
    const int32_t t = f.ns_row[row];
    int lo = 0, hi = *f.n_tags;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (f.tags[mid] < t) lo = mid + 1;
        else hi = mid;
    }
    if (lo < *f.n_tags && f.tags[lo] == t) return fmaxf(floor_, f.tag_floor[lo]);
    return INFINITY;
}
// nf: the per-namespace floors, or NULL (one floor for all rows)
cudaError_t launch_split_flags(const HopPlan &p, const float *row_ub, const float *floor_p,
                               const NsFloors *nf, int32_t *split_skip, int32_t *slot_skip,
                               int32_t *kept_rows, int64_t *kept_count, int32_t *kept_segs,
                               KeptScratch &ks, cudaStream_t st, int *launches);
// The floors of a scoped batch: tags = the distinct q_ns of the n_real query
// columns, and for each tag the largest of (a) the smallest score that the
// filter bound of any of its queries admits and (b) the k-th largest lb over
// the split rows of that namespace, taken heaviest first (split_order), at
// most PF_ROWS of them (any subset of a namespace's rows gives a floor that
// each of its queries' k-th largest final score reaches).
cudaError_t launch_ns_floors(const unsigned long long *bound, const int32_t *q_ns, int n_real,
                             const float *lb, const int32_t *ns_row, const int32_t *split_row,
                             const int32_t *split_order, int64_t n_split, int k, int32_t *tags,
                             int *n_tags, float *tag_floor, cudaStream_t st);
// floor = max(the smallest score any real column's filter bound admits,
// and, if lb_rows != NULL, the k-th largest lb over the rows
// lb_rows[order[i]], i < n_lb_rows), written to floor_out.  The second term
// is only valid when every row may be selected by every query (no namespace
// scope).
cudaError_t launch_prune_floor(const unsigned long long *bound, int n_real, const float *lb,
                               const int32_t *lb_rows, const int32_t *order, int64_t n_lb_rows,
                               int k, float *floor_out, cudaStream_t st);
cudaError_t launch_fill_f32(float *v, int64_t n, float x, cudaStream_t st);

// ------------------------------------------------------------------ reach (ak_reach.cu)
// Final scores of a few candidate rows straight from u: s^(H)_j = u_j +
// sum_t alpha^t sum_k C_t[k][j] u_k with graph-only reach coefficients.
constexpr int REACH_T = 128;         // candidate rows kept
struct ReachBuild {
    int64_t n, n_split;
    int H;
    const int32_t *split_row, *split_order;
    const float *mup;                // mass levels [H + 1][n] (candidate choice)
    const int64_t *in_ptr;           // in-edge CSR (row space)
    const int32_t *in_src;
    const float *in_w;
    const int64_t *row_ptr;          // out-edge CSR (chunk IDs)
    const int32_t *col, *row_of;
    const float *w;
    int32_t *rows;                   // [REACH_T] candidate rows
    int *t_cnt;                      // their number (device)
    int32_t *map;                    // [n] row -> candidate slot or -1
    float *C;                        // [H][n][REACH_T]
};
cudaError_t launch_reach_build(const ReachBuild &rb, cudaStream_t st);
// The reach path's floor, flags and plan, without the per-row bound arrays:
// floor = the k-th largest lower bound over the (up to 1024) heaviest split
// rows, computed for those rows only; then every row's upper bound against
// it: keep[REACH_T] flags the candidates that reach it, *bad counts the
// other rows that do, and the last CTA to finish writes the plan
// (REACH_PLAN_INTS below).  ws: int32[REACH_T + 2] scratch (keep, bad, done).
struct ReachFlags {
    const float *u0, *l0;            // u's row maxima / minima [n]
    const float *mup, *mdn;          // mass levels [H + 1][n]
    const unsigned int *ext;         // Umax / Lmin (launch_final_bounds' encoding)
    int64_t n;
    int H;
    float alpha;
    const int32_t *split_row, *split_order;
    int64_t n_lb;                    // heaviest split rows taken for the floor (<= 1024)
    int k;
    const int32_t *map;              // row -> candidate slot or -1
    const int *t_cnt;                // candidates (device)
    float *floor_out;
    int32_t *ws;
    int32_t *plan;                   // [REACH_PLAN_INTS]
};
cudaError_t launch_reach_flags(const ReachFlags &f, cudaStream_t st, int *launches);
int reach_parts();                   // CTAs of the candidates' pass (partial rows)
// The call's plan on the device (int32[REACH_PLAN_INTS], written by
// launch_reach_flags): plan[0] = 1 when the flagged candidates suffice for
// top-k (else the hops run), plan[1] = their number nk, plan[2..] their
// slots in ascending order, plan[REACH_PLAN_WIDE] = 1 when a flagged slot
// is 64 or above.
constexpr int REACH_PLAN_WIDE = REACH_T + 2;
constexpr int REACH_PLAN_INTS = REACH_T + 3;
// Rows of the packed coefficients: n rounded up to a whole 64-row stage.
int64_t reach_pad_rows(int64_t n);
// Every candidate's combined coefficients sum_t alpha^t C_t as bf16 hi + lo,
// [REACH_T][reach_pad_rows(n)] each (graph-only; repacked when the graph,
// alpha or H change).
cudaError_t launch_reach_pack(const float *C, int64_t n, int H, float alpha, uint16_t *coef_hi,
                              uint16_t *coef_lo, cudaStream_t st);
// partial: [reach_parts()][REACH_T][bp] scratch; with plan[0] = 1 the
// flagged candidates' keys are written to each real column's buffer
// (cnt[b] = nk); with plan[0] = 0 both kernels return at once.  bp = 128
// or 256.  u_hi, u_lo: the score GEMM's split-bf16 u, [n][bp] each.
cudaError_t launch_reach_scores(const uint16_t *u_hi, const uint16_t *u_lo, int bp, int B,
                                int64_t n, const uint16_t *coef_hi,
                                const uint16_t *coef_lo, const int32_t *plan, const int32_t *rows,
                                const int32_t *ext_of, float *partial, unsigned int *cnt,
                                unsigned long long *buf, int64_t cap, int *status, cudaStream_t st,
                                int *launches);
// slot_split[s] = r for every partial slot s of split row r.
cudaError_t launch_slot_owner(const int64_t *split_slot0, int64_t n_split, int32_t *slot_split,
                              cudaStream_t st);
// `counters` = 2 device ints, zeroed by the launcher (work queues).
// `flt` may be NULL (no filter), `hb` NULL (no row bounds).
cudaError_t launch_hop(const HopPlan &p, const float *u, const float *in, float *out, int bp,
                       float alpha, float *partial, int *counters, const HopFilter *flt,
                       cudaStream_t st, int *launches, const HopBound *hb = nullptr);

// ------------------------------------------------------------------ selection
// Top-k of every column of a slab (a3): bound from a row sample, filter
// pass, merge (see ak_select.cu).  The workspace holds sp.words 64-bit words.
struct SelectPlan {
    int64_t n;          // rows
    int bp, k;
    int64_t stride;     // sample every stride-th row
    int64_t n_sample;
    int64_t cap;        // buffer capacity per column
    // workspace offsets in 64-bit words: bounds, counts, buffers, the
    // sample transposed to [bp][n_sample] 32-bit keys
    int64_t off_bound, off_cnt, off_buf, off_tr, words;
};
// force_stride > 0 samples every force_stride-th row instead of the default.
SelectPlan select_plan(int64_t n, int bp, int k, int sm_count, int64_t force_stride = 0);

// Retrieval: rows are store rows; keys and outputs carry chunk IDs
// (ext_of), so ties resolve to the lower chunk ID; page_row is indexed by
// row (row_of).  Scores are divided by Z = sum of zpart's first n_ztiles rows.
// With a scope (ns.q_ns != NULL) a query whose namespace holds fewer than k
// chunks gets its list padded with ID -1, score 0, page -1; with
// sort_by_time the k winners are written in ascending chunk ID order
// (Algorithm 1, SortByTime) instead of by score.
cudaError_t launch_select(const SelectPlan &sp, const float *s, int b, unsigned long long *ws,
                          const float *zpart, int64_t n_ztiles, const int32_t *ext_of,
                          const int32_t *row_of, const int32_t *page_row, int64_t *ids,
                          float *scores, int32_t *page_ids, int32_t *n_pages, int *status,
                          NsScope ns, int sort_by_time, cudaStream_t st, int *launches);
// Same selection over signed values (cosines) among rows whose chunk ID is
// below id_limit: the k best of each of the b columns go to nbr_ids /
// nbr_cos rows c_base .. c_base+b-1.
cudaError_t launch_select_signed(const SelectPlan &sp, const float *s, int b,
                                 unsigned long long *ws, const int32_t *ext_of, int64_t id_limit,
                                 int64_t c_base, int32_t *nbr_ids, float *nbr_cos, int *status,
                                 cudaStream_t st, int *launches, NsScope ns = NsScope{});
// Bound pass alone over signed values: bound[c] for the b real columns
// (the k-th largest sampled key; padding columns get an all-ones bound).
// Bound only, unsigned keys (retrieval): ws + sp.off_bound gets the bound,
// the column counts are cleared.  For a filter fused into the last hop or
// into the score.  `slack` lowers each bound by that many units of the
// score's last place (margin for a sample computed by another launch).
cudaError_t launch_sample_bound(const SelectPlan &sp, const float *s, int b,
                                const int32_t *ext_of, unsigned long long *ws, cudaStream_t st,
                                int *launches, uint32_t slack = 0, NsScope ns = NsScope{});
// A column of the last hop recomputed by the merge when the filter fused
// into that hop (which writes no output slab) overflowed its buffer:
// dst[j,c] = u[j,c] + alpha * sum_{e in in(j)} in_w[e] * prev[in_src[e],c].
// Without hops (the score itself, fused with the filter, wrote no slab):
// dst[j,c] = exp(tau <e_j, q_c> - shift[c]) from the stored bf16 values.
struct ColumnRecompute {
    int kind;     // 0 none, 1 last hop, 2 score
    const float *u, *prev;
    const int64_t *in_ptr;
    const int32_t *in_src;
    const float *in_w;
    float alpha;
    const uint16_t *emb, *qp;   // kind 2: E [n][dim], padded queries [bp][dim]
    int dim;
    float tau;
    const float *shift;
    float *dst;   // [n][bp]; the merge reads the overflowed column from here
};
// Row j -> chunk ID of a strided sample: out[v] = ext_of[v * stride].
cudaError_t launch_ext_sample(const int32_t *ext_of, int64_t n_sample, int64_t stride,
                              int32_t *out, cudaStream_t st);
// Merge only: the k winners per column from the buffers filled by a filter
// pass (falls back to the column of `s` where a buffer overflowed, after
// recomputing it into s when `rc` is given; then s must be rc->dst).
cudaError_t launch_topk_merge(const SelectPlan &sp, const float *s, int b,
                              const unsigned long long *ws, const float *zpart, int64_t n_ztiles,
                              const int32_t *ext_of, const int32_t *row_of,
                              const int32_t *page_row, int64_t *ids, float *scores,
                              int32_t *page_ids, int32_t *n_pages, int *status,
                              const ColumnRecompute *rc, NsScope ns, int sort_by_time,
                              cudaStream_t st, int *launches);
cudaError_t launch_sample_bound_signed(const SelectPlan &sp, const float *s, int b,
                                       const int32_t *ext_of, int64_t id_limit,
                                       unsigned long long *ws, unsigned long long *bound,
                                       cudaStream_t st, int *launches, NsScope ns = NsScope{});
// bound[c] = the k-th largest of the n_sample keys keys_t[c][*] (k <= 64) as a
// key with the chunk-ID half zero, 0 if fewer than k keys are nonzero; ~0
// for the padding columns b <= c < bp; cnt[c] = 0.  One CTA a column.
cudaError_t launch_sample_kth_keys(const uint32_t *keys_t, int64_t n_sample, int bp, int b, int k,
                                   unsigned long long *bound, unsigned int *cnt, cudaStream_t st,
                                   int *launches);
// Top-k of each column's filter buffer (no overflow): nbr rows 0..n_cols-1.
cudaError_t launch_buf_merge_signed(const unsigned int *cnt, const unsigned long long *buf,
                                    int64_t cap, int64_t n_cols, int k, int32_t *nbr_ids,
                                    float *nbr_cos, int *status, cudaStream_t st, int *launches);

}  // namespace ak
