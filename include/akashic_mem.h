/*
 * akashic_mem.h -- C ABI of the GB300 (sm_103a) memory-retrieval library.
 *
 * The library keeps a chunked memory store on one GPU and runs the
 * data-parallel hot path of MemAttention's memory system (arXiv 2607.05708)
 * in its Dense-only form (embedding similarity in place of the LLM matcher,
 * §5.5):
 *
 *   retrieve  score every chunk against a batch of queries (softmax over
 *             chunks), spread the scores along the cross-chunk relation
 *             graph, keep the top-k chunks per query and resolve them to the
 *             pages that hold them (query-aware retrieval, §4.1 and
 *             Algorithm 1's retrieval steps; the locality gap |P(R_t)|,
 *             §3.2);
 *   append    add immutable chunk records, each with a logical ID and a
 *             physical page (§4.2: logical identity is separate from
 *             physical placement);
 *   update    for new chunks, select the top-M related prior chunks by
 *             cosine similarity and link them both ways in the relation
 *             graph (cross-chunk selection, §4.1 and Algorithm 1's
 *             LLMSelect of related prior chunks).
 *
 * Conventions
 *   - Every entry point returns an akashic_status_t and never throws.
 *     akashic_mem_last_error() gives a thread-local message for the last
 *     failure on the calling thread.
 *   - The library owns all store memory; the caller owns every argument
 *     buffer.  Array arguments named "device" are CUDA device pointers on
 *     the store's device; "host" ones are host pointers.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Calls are stream-ordered: device inputs may be reused once
 *     the stream has passed the call; outputs are valid once it has
 *     completed.  Faults found by a kernel (a bounded device wait that
 *     expired, an index out of range) are recorded in a device status word
 *     and returned by the next akashic_mem_sync() on that store.
 *   - retrieve may run concurrently on different streams (each stream gets
 *     its own scratch); append and update must not overlap any other call
 *     on the same store.
 *   - Embeddings are bf16, passed as their raw 16-bit patterns (uint16_t),
 *     row-major, `dim` values per row.
 */
#ifndef AKASHIC_MEM_H
#define AKASHIC_MEM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct akashic_mem akashic_mem_t; /* opaque, library-owned */

typedef enum {
    AKASHIC_OK = 0,
    AKASHIC_EINVAL = 1,    /* bad argument (see each call)                       */
    AKASHIC_ENOMEM = 2,    /* a device or host allocation failed                 */
    AKASHIC_ECAPACITY = 3, /* the store's chunk capacity would be exceeded       */
    AKASHIC_ECUDA = 4,     /* a CUDA runtime/driver call failed                  */
    AKASHIC_ETIMEOUT = 5,  /* a bounded device-side wait expired                 */
    AKASHIC_EDEVICE = 6,   /* a kernel found an inconsistent index or size       */
    AKASHIC_ERANGE = 7     /* scores would leave fp32 range (see retrieve)       */
} akashic_status_t;

/* Largest hop count retrieve accepts. */
#define AKASHIC_MAX_HOPS 16

typedef struct {
    int32_t dim;             /* embedding width; multiple of 64, 64..4096          */
    int64_t capacity;        /* maximum number of chunks, 1..2^31-1                */
    int32_t chunks_per_page; /* page packing for appends given no page table (>=1) */
    int32_t device;          /* CUDA device ordinal                                */
    float temperature;       /* softmax temperature tau; 0 => 1/sqrt(dim)          */
    float relation_scale;    /* edge logit = scale * cosine in updates; 0 => 10    */
} akashic_mem_config_t;

/* Create an empty store on cfg->device.  Allocates the embedding table
 * (capacity x dim bf16) and the page table up front; the relation graph
 * grows on demand.  EINVAL for an out-of-range field, ENOMEM if the device
 * cannot hold the table. */
akashic_status_t akashic_mem_create(const akashic_mem_config_t *cfg, akashic_mem_t **out);

/* NULL-safe.  Synchronises the store's device and frees everything. */
void akashic_mem_destroy(akashic_mem_t *m);

/* Append n immutable chunk records (§4.2: chunks are written once; the
 * store's IDs are assigned in append order, first_id .. first_id+n-1).
 * In device memory the batch is laid out in page order (ID order within a
 * page), so that chunks the placement co-locates are adjacent rows; IDs
 * are unaffected.
 *   emb      device, n x dim bf16 bits, 16-byte aligned.
 *   page_of  device int32[n], the physical page of each new chunk (>= 0), or
 *            NULL: fresh pages after the highest page in use, packed
 *            chunks_per_page at a time in ID order.
 *   row_ptr, col, aff  optional initial out-edges of the NEW rows, as a CSR
 *            over their local rows: row_ptr device int64[n+1] (row_ptr[0]
 *            may be non-zero; offsets index col/aff), col device int32
 *            (global target IDs < first_id+n, never the row itself, strictly
 *            ascending within a row), aff device float (edge logits; the
 *            relation weight of an edge is the softmax of its row's logits).
 *            row_ptr NULL => no edges (col and aff must then be NULL too);
 *            col and aff may be NULL when row_ptr describes no edges.
 *   first_id_out  host, receives first_id (may be NULL).
 * ECAPACITY if the store would exceed its capacity; EINVAL on a bad
 * argument; EDEVICE (at once, since this call synchronises) if the edges
 * are not a valid CSR.  Synchronises `stream`. */
akashic_status_t akashic_mem_append_chunks(akashic_mem_t *m, const uint16_t *emb, int64_t n,
                                           const int32_t *page_of, const int64_t *row_ptr,
                                           const int32_t *col, const float *aff,
                                           int64_t *first_id_out, void *stream);

/* Relation update for the chunks [first, first+n) (cross-chunk selection,
 * Algorithm 1's LLMSelect of related prior chunks, in its dense form): for
 * each such chunk c, its top-M
 * prior chunks j < first by cosine <e_c, e_j> of the stored bf16 values
 * (no further normalisation), ordered by cosine descending then lower ID,
 * become its out-edges with logit relation_scale * cos; with reciprocal != 0
 * each chosen j also gets the edge j -> c with the same logit.  Rows stay
 * sorted by column and every touched row's weights are re-normalised (row
 * softmax).  New chunks are not linked to each other.
 * EINVAL if first+n > size, M < 1, M > 64, M > first, or any row in
 * [first, first+n) already has out-edges; EDEVICE if an existing edge
 * already points into [first, first+n).  Synchronises `stream`. */
akashic_status_t akashic_mem_update_relations(akashic_mem_t *m, int64_t first, int64_t n,
                                              int32_t M, int32_t reciprocal, void *stream);

/* Query-aware retrieval (§4.1, Algorithm 1's retrieval steps, Dense-only form):
 *   z[b,i] = tau <q_b, e_i>;  s0[b,:] = softmax over chunks of z[b,:];
 *   s^(0) = u = exp(z - c_b);  s^(h)_j = u_j + alpha sum_{i->j} w_ij s^(h-1)_i
 *   for h = 1..hops (mass flows along out-edges i -> j);
 *   score_j = s^(hops)_j / sum_i u_i.
 * Per query the k chunks with the largest score, ordered by score descending
 * then lower chunk ID, and their pages (FetchByID; the number of distinct
 * pages is |P(R_t)| of §3.2).
 *   q        device, B x dim bf16 bits.
 *   ids      device int64[B*k]   (row b holds query b's winners)
 *   scores   device float[B*k]   (the final scores above)
 *   page_ids device int32[B*k]   (page_of of each winner; may be NULL)
 *   n_pages  device int32[B]     (distinct pages per query; may be NULL)
 * hops = 0 or alpha = 0 => plain top-k of the softmax.  The shift c_b is the
 * bound tau |q_b| max_i |e_i|, so no extra pass is needed; ERANGE (via
 * akashic_mem_sync) if 2 c_b > 80, where exp would leave fp32 range.
 * EINVAL if B < 1, k < 1, k > 64, k > size, hops < 0, hops > 16, alpha < 0
 * or not finite.
 * Does not synchronise, with one exception: with hops = 2, alpha > 0, no
 * scope and 65 to 256 queries in a batch of 128 or 256, the host waits once
 * per batch for the device's decision between the two-hop path from reach
 * coefficients and the hops (an event recorded after a 12-byte copy, not the
 * whole stream; the candidates' pass is already queued behind it, so the
 * GPU does not idle); the first such call after the graph changed also waits
 * while it builds their graph-only tables.
 * Graph-only tables built by a call on one stream are waited for (an event,
 * not a host wait) by calls on every other stream. */
akashic_status_t akashic_mem_retrieve(akashic_mem_t *m, const uint16_t *q, int32_t B, int32_t k,
                                      float alpha, int32_t hops, int64_t *ids, float *scores,
                                      int32_t *page_ids, int32_t *n_pages, void *stream);

/* Namespace tags (§4.1: memory chunks are keyed by (user_id, session_id),
 * which isolate tenants and sessions).  The caller maps each (user_id,
 * session_id) pair to one int32 tag; ns (device int32[n]) sets the tags of
 * chunk IDs [first, first+n).  Every chunk starts with tag 0.
 * EINVAL if the range leaves the store or ns is NULL with n > 0.
 * Stream-ordered, does not synchronise. */
akashic_status_t akashic_mem_set_namespace(akashic_mem_t *m, int64_t first, int64_t n,
                                           const int32_t *ns, void *stream);

/* Delete chunks (the deletions of cross-chunk compaction, Algorithm 1
 * JointCompact / "Apply updates U and deletions D"; stale copies are
 * logically tombstoned, §4.2).  ids: device int64[n] chunk IDs.  A deleted
 * chunk keeps its ID and row but gets no score (it adds nothing to Z or to
 * propagation), is never selected by retrieval and never chosen by a
 * relation update; every relation edge into or out of it is dropped and the
 * rows that lost edges are re-softmaxed; the in-edge transpose and the hub
 * plan are compacted to match.  Deleting a chunk twice is harmless.  A later
 * append may not pass edges that point at a deleted chunk (EDEVICE).
 * EINVAL if n < 0, ids is NULL with n > 0, or any ID lies outside
 * [0, size) (then nothing changes).  Synchronises `stream`. */
akashic_status_t akashic_mem_delete(akashic_mem_t *m, const int64_t *ids, int64_t n,
                                    void *stream);

/* Memory Manager (§4.2, Algorithm 2), on the page directory (page_of).
 * The model calls have dense stand-ins: co-retrieval statistics over the
 * requests passed in (sel(c) = requests that retrieved c, co(a, b) = those
 * that retrieved both); affinity(a, b) = co / (sel(a) + sel(b) - co), "high
 * association" when co >= tau_assoc * (sel(a) + sel(b) - co) (fp64, tau
 * rounded to fp32; the paper's tau_assoc is 0.7, §5.5).
 *
 * Relocation (Algorithm 2: LLMCoLocate, then PackIntoNewBlocks of the
 * time-sorted group and MarkInvalid of the old copies).
 *   S  device int64[n_req][s_len], the retrieved chunk IDs per request
 *      (-1, IDs outside the store, deleted chunks and repeats are
 *      skipped), 1 <= s_len <= 64.
 * The batch's statistics are added first; then, request by request, the
 * chunks of the request that are highly associated with another of its
 * chunks (LLMCoLocate), if two or more and not all on one page, are written
 * out of place in chunk-ID order (SortByTime) into fresh pages of
 * chunks_per_page slots; each old copy becomes an invalid slot of its page.  Synchronises `stream`.
 * EINVAL on bad sizes or tau outside [0, 1]. */
akashic_status_t akashic_mem_relocate(akashic_mem_t *m, const int64_t *S, int32_t n_req,
                                      int32_t s_len, float tau_assoc, void *stream);

/* Block compaction (Algorithm 2: LiveChunks, PartitionByUserSession,
 * LLMGroup, PackIntoNewBlocks, Release; phi(B) of §4.2): every page
 * whose invalid ratio phi = (slots - live) / slots is >= theta (0.75 in the
 * paper) is compacted: its live chunks are partitioned by namespace
 * (akashic_mem_set_namespace), grouped within a partition by the connected
 * components of highly associated pairs (LLMGroup), and repacked into fresh
 * pages partition by partition, group by group (groups by earliest chunk
 * ID), chunk ID order within a group; the page is released.  *released
 * (may be NULL) = pages released.  Synchronises `stream`.
 * EINVAL if theta is outside (0, 1] or tau outside [0, 1]. */
akashic_status_t akashic_mem_compact_pages(akashic_mem_t *m, float theta, float tau_assoc,
                                           int64_t *released, void *stream);

/* Page accounting, host int64 out[5]: pages in use, slots in use (live and
 * invalid), live slots, chunk writes (appends + relocations + compaction
 * moves), chunks appended.  Space amplification = out[1] / out[2]; write
 * amplification = out[3] / out[4].  Synchronises the device. */
akashic_status_t akashic_mem_page_stats(akashic_mem_t *m, int64_t *out);

/* page_of: device int32[size]: the page of every chunk ID (the directory
 * retrieval resolves through).  Stream-ordered. */
akashic_status_t akashic_mem_export_pages(akashic_mem_t *m, int32_t *page_of, void *stream);

/* Retrieval scoped to the caller's namespace, with optional chronological
 * order (§4.1: candidates are the chunks of the current user_id/session_id;
 * Algorithm 1's SortByTime: the selected chunks are returned in time
 * order).  As akashic_mem_retrieve, except:
 *   q_ns          device int32[B] or NULL: query b selects only among chunks
 *                 whose tag equals q_ns[b] (scores, Z and propagation are
 *                 those of the whole store; the scope applies to the
 *                 candidates).  A namespace with fewer than k chunks pads
 *                 the query's list with ID -1, score 0, page -1, and
 *                 n_pages counts the real entries only.
 *   sort_by_time  != 0: the k selected chunks are written in ascending chunk
 *                 ID (IDs are assigned in append order) instead of by score.
 * Errors as akashic_mem_retrieve.  With q_ns given it does not synchronise;
 * with q_ns NULL it may wait on `stream` as akashic_mem_retrieve does. */
akashic_status_t akashic_mem_retrieve_scoped(akashic_mem_t *m, const uint16_t *q, int32_t B,
                                             int32_t k, float alpha, int32_t hops,
                                             const int32_t *q_ns, int32_t sort_by_time,
                                             int64_t *ids, float *scores, int32_t *page_ids,
                                             int32_t *n_pages, void *stream);

/* Read back the canonical out-edge CSR.  With all array pointers NULL only
 * the sizes are returned (host n_rows, host nnz).  Otherwise row_ptr device
 * int64[n_rows+1], col device int32[nnz], and optionally aff / w device
 * float[nnz] (edge logits and row-softmax weights) are written.
 * Synchronises `stream`. */
akashic_status_t akashic_mem_export_csr(akashic_mem_t *m, int64_t *n_rows, int64_t *nnz,
                                        int64_t *row_ptr, int32_t *col, float *aff, float *w,
                                        void *stream);

/* Number of chunks in the store and the relation graph's edge count (host). */
akashic_status_t akashic_mem_size(const akashic_mem_t *m, int64_t *n_chunks, int64_t *nnz);

/* Synchronise `stream`, then return and clear the store's device status
 * word (ETIMEOUT, EDEVICE or ERANGE from an earlier kernel), else OK. */
akashic_status_t akashic_mem_sync(akashic_mem_t *m, void *stream);

/* Phase timing.  With profiling on, each call records CUDA events on its
 * own stream around every phase; akashic_mem_phase_times synchronises the
 * recorded events and returns, per phase, the summed device milliseconds
 * and the number of kernel launches since the last reset, then resets.
 * Phases: */
enum {
    AKASHIC_PHASE_SCORE = 0,     /* query x chunk score GEMM + exp + Z partials */
    AKASHIC_PHASE_PROPAGATE = 1, /* relation-graph hops                         */
    AKASHIC_PHASE_SELECT = 2,    /* top-k candidates, merge, page resolve       */
    AKASHIC_PHASE_RELATE = 3,    /* new x store cosine GEMM + top-M             */
    AKASHIC_PHASE_GRAPH = 4,     /* CSR insert, weights, transpose rebuild      */
    AKASHIC_PHASE_RELOCATE = 5,  /* co-retrieval counts + relocation            */
    AKASHIC_PHASE_COMPACT = 6,   /* block compaction                            */
    AKASHIC_PHASE_BOUND = 7,     /* last hop's row bounds, floor and skip flags */
    AKASHIC_PHASE_LAST_HOP = 8,  /* last hop with the top-k filter fused        */
    /* three parts of AKASHIC_PHASE_GRAPH in a relation update, also counted
     * in it: */
    AKASHIC_PHASE_CSR_INSERT = 9,  /* new CSR: old rows moved, new rows and
                                      reciprocal edges placed                 */
    AKASHIC_PHASE_TRANSPOSE = 10,  /* row softmax and the in-edge transpose   */
    AKASHIC_PHASE_HUB_PLAN = 11,   /* the hop's hub segment plan rebuilt      */
    AKASHIC_PHASE_COUNT = 12
};
akashic_status_t akashic_mem_set_profiling(akashic_mem_t *m, int32_t on);
akashic_status_t akashic_mem_phase_times(akashic_mem_t *m, float *ms, int32_t *launches);

/* Softmax scores for callers that cannot allocate device memory.
 *
 * The paper has no counterpart: this is a library convenience.  A serving
 * runtime that works inside a memory pool it reserved up front, code that
 * is recording a stream capture, or a host without a device allocator
 * cannot call cudaMalloc when it needs scores, and akashic_mem_create
 * allocates.  This
 * call needs no store and allocates nothing: it computes, over caller-owned
 * buffers, the score step of retrieval
 *   u[j*B + b] = exp(tau <e_j, q_b> - c_b),   z[b] = sum_j u[j*B + b],
 *   c_b = tau |q_b| max_j |e_j|,
 * so that u[:, b] / z[b] is the softmax over the n chunks (the same kernel
 * as the score step of akashic_mem_retrieve).
 *   emb    device, n x dim bf16 bits (chunk j in row j), 16-byte aligned
 *   q      device, B x dim bf16 bits, 16-byte aligned
 *   B      32, 64, 128 or 256 (pad with zero queries); larger B is rejected
 *          because the fixed scratch holds at most 256 queries
 *   temperature  tau; 0 => 1/sqrt(dim)
 *   u      device float[n*B] (output, chunk-major), 16-byte aligned
 *   z      device float[B] (output)
 *   shift  device float[B] (output c_b) or NULL
 *   status device int32 (output) or NULL: 0, or ERANGE / ETIMEOUT found by
 *          the kernels
 * Its scratch is a fixed 320 KiB array in device memory, present on every
 * GPU that runs this call until the process exits (no allocation ever
 * happens).  The first call on a device does a one-time set-up while the
 * device is current: it looks up that array's address with
 * cudaGetSymbolAddress and sets the score kernel's shared-memory limit for
 * all four widths B; make that first call before capturing a stream.  Every call shares the array, so calls whose
 * work overlaps on the GPU (different streams without ordering) race and
 * must not be issued.  Stream-ordered; does not synchronise.
 * EINVAL for a NULL pointer, misalignment, n < 1, dim outside [64, 4096]
 * or not a multiple of 64, B not in {32, 64, 128, 256}, or a device with
 * more than 256 SMs; ECUDA if a launch fails. */
akashic_status_t akashic_mem_softmax_scores_noalloc(const uint16_t *emb, int64_t n, int32_t dim,
                                                    const uint16_t *q, int32_t B,
                                                    float temperature, float *u, float *z,
                                                    float *shift, int32_t *status, void *stream);

/* Check of the failure path of the bounded device waits.  The paper has no
 * counterpart: this is a library self-test.  Every wait inside the library's
 * kernels (on a barrier, a copy, a peer's flag) gives up after a bounded number
 * of polls, records ETIMEOUT in the store's status word and lets its kernel
 * return, so a fault shows up as an error code and the context stays usable.
 * This call launches one thread that waits, with that same wait, for a barrier
 * phase that nothing ever completes, and gives up after `polls` polls (the
 * kernels' waits allow 2^26).  The next akashic_mem_sync() on `stream` then
 * returns ETIMEOUT and clears the word; the store is otherwise untouched.
 * Stream-ordered; does not synchronise.  EINVAL for a NULL store or polls
 * outside [1, 2^26]. */
akashic_status_t akashic_mem_check_wait_timeout(akashic_mem_t *m, uint32_t polls, void *stream);

/* Stable sort of n (key, value) pairs of 32-bit words in device memory of the
 * current device, by the low `bits` bits of the keys (pairs with equal low
 * bits keep their input order), in place: keys[i] and vals[i] travel
 * together.  The paper has no counterpart: this is the sort primitive that the
 * library's own steps use (the in-edge transpose of the relation CSR, the
 * reciprocal edges of a relation update, the hub plan of the propagation
 * hop), exported so that it can be checked on its own.  Allocates and frees
 * its scratch (2n words and the digit histograms) and synchronises `stream`.
 * EINVAL for n < 0, n > 2^31 - 1, NULL buffers with n > 1, or bits outside
 * [0, 32]; ENOMEM if the scratch cannot be allocated; ECUDA if a launch fails.
 * n <= 1 or bits = 0 leaves the buffers untouched. */
akashic_status_t akashic_mem_sort_pairs(uint32_t *keys, uint32_t *vals, int64_t n, int32_t bits,
                                        void *stream);

/* Thread-local description of the last failure on this thread ("" if none). */
const char *akashic_mem_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* AKASHIC_MEM_H */
