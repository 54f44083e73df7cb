/*
 * Akashic MemAttention, dense surrogate -- CPU ORACLE.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load this library.  The product path
 * (the CUDA library) never calls it and shares no code with it.
 *
 * Plain, slow, single-threaded C.  Every quantity is computed in IEEE fp64
 * from the stored bf16 values (widened exactly), with plain loops in index
 * order, libm exp(), and qsort for ordering.  Nothing is blocked, fused or
 * reordered beyond what the definitions below state.
 *
 * What it computes (arXiv 2607.05708; the paper's own matching is an LLM
 * call, LLMSelect in Algorithm 1, §4.1; its Dense-only ablation, §5.5,
 * replaces that call by embedding similarity, which is the form written out
 * here):
 *
 *  Score (query-aware retrieval, §4.1, Algorithm 1 retrieval half):
 *      z[b,i] = tau * <q_b, e_i>,  u[b,i] = exp(z[b,i] - c_b),
 *      Z_b = sum_i u[b,i],  s0 = u / Z  (a softmax over chunks),
 *      c_b = max_i z[b,i]  (any shift gives the same s0; this one is exact).
 *  Propagate along the cross-chunk relation graph (the semantic relations
 *      across chunks that cross-chunk inference recovers, §4.1):
 *      s^(0) = u;  s^(h)_j = u_j + alpha * sum_{i -> j} w_ij * s^(h-1)_i,
 *      h = 1..H, with w_ij the row softmax of the edge logits of row i.
 *      Final score  s_j = s^(H)_j / Z_b  (not renormalised).
 *      The sum is taken by SCATTERING over out-edges, source by source.
 *  Top-k: the k chunks with the largest final score, ordered by score
 *      descending, then by lower chunk ID (the top-p selection of §4.1).
 *  Page resolve (FetchByID, Algorithm 1; the locality gap |P(R_t)|, §3.2):
 *      page_ids = page_of[ids], n_pages = number of distinct page IDs.
 *
 *  Relation update (cross-chunk selection of related prior chunks for a new
 *      chunk, Algorithm 1 compaction half, §4.1):
 *      cos(n, i) = <e_n, e_i> over the stored bf16 values (no further
 *      normalisation) for every prior chunk i < first; keep the top-M by
 *      (cos descending, lower ID); new row n gets those M columns in
 *      ascending order with logit scale * cos; with `reciprocal`, each chosen
 *      j also gets the edge j -> n with the same logit.  Rows stay sorted by
 *      column; the weights of every row are the row softmax of its logits.
 *
 *  Namespace-scoped retrieval (the candidate set is the chunk table T[u][s]
 *      of the caller's (user_id, session_id), §4.1 and Algorithm 1 retrieval
 *      half) and SortByTime (Algorithm 1: the selected chunks are returned in
 *      chronological order):  every chunk carries a namespace tag ns_of[i];
 *      query b selects only among chunks with ns_of[i] == q_ns[b] (scores,
 *      Z and propagation are those of the whole store; the scope applies to
 *      the candidates); with fewer than k such chunks the list is padded
 *      with ID -1, score 0, page -1.  With sort_by_time the selected IDs
 *      are reordered by ascending chunk ID (IDs are assigned in append
 *      order), padding last.
 *
 *  Deletion (JointCompact's deletions D applied to the chunk table,
 *      Algorithm 1; invalidated copies are logically tombstoned, §4.2): a
 *      deleted chunk is no longer part of the store's memory: it gets no
 *      score (u = 0, so it adds nothing to Z or to propagation) and is never
 *      selected; every relation edge into or out of it is dropped and the
 *      weights of the rows that lost edges are the row softmax of what
 *      remains.
 *
 * Readings where the paper is silent (also recorded in the design notes):
 *   - temperature tau defaults to 1/sqrt(dim) for every store;
 *   - multi-hop form s^(h) = u + alpha * s^(h-1) R (truncated personalised
 *     PageRank series), mass flows along out-edges i -> j, no renormalisation;
 *   - ties in score resolve to the lower chunk ID;
 *   - reciprocal edges never evict: old rows grow past M out-edges;
 *   - new chunks are linked only to prior chunks, not to each other.
 *
 * Return codes: 0 ok, 1 invalid argument, 2 out of memory.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORA_OK 0
#define ORA_EINVAL 1
#define ORA_ENOMEM 2

static double bf16_widen(uint16_t h)
{
    uint32_t bits = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

/* ------------------------------------------------------------ relation weights */

/* w_e = exp(aff_e - max_row) / sum_row exp(aff_f - max_row), row by row. */
int ora_row_softmax(int64_t n_rows, const int64_t *row_ptr, const float *aff, double *w)
{
    if (n_rows < 0 || !row_ptr)
        return ORA_EINVAL;
    for (int64_t i = 0; i < n_rows; ++i) {
        int64_t a = row_ptr[i], b = row_ptr[i + 1];
        if (b <= a)
            continue;
        double m = -INFINITY;
        for (int64_t e = a; e < b; ++e)
            if ((double)aff[e] > m)
                m = (double)aff[e];
        double sum = 0.0;
        for (int64_t e = a; e < b; ++e) {
            w[e] = exp((double)aff[e] - m);
            sum += w[e];
        }
        for (int64_t e = a; e < b; ++e)
            w[e] /= sum;
    }
    return ORA_OK;
}

/* ------------------------------------------------------------ ordering */

typedef struct {
    double key;
    int64_t id;
} ora_pair;

/* score descending, then ID ascending */
static int cmp_desc_id(const void *pa, const void *pb)
{
    const ora_pair *a = (const ora_pair *)pa, *b = (const ora_pair *)pb;
    if (a->key > b->key)
        return -1;
    if (a->key < b->key)
        return 1;
    return (a->id < b->id) ? -1 : (a->id > b->id);
}

static int cmp_i64(const void *pa, const void *pb)
{
    int64_t a = *(const int64_t *)pa, b = *(const int64_t *)pb;
    return (a < b) ? -1 : (a > b);
}

/* ------------------------------------------------------------ retrieve */

/*
 * emb      n x dim bf16 bits, chunk i in row i
 * q        n_q x dim bf16 bits
 * row_ptr  n+1, col nnz, w nnz (out-edge CSR, w from ora_row_softmax); may be
 *          NULL when hops == 0
 * page_of  n (may be NULL: page outputs are then skipped)
 * outputs  ids[n_q*k], scores[n_q*k] (final s), page_ids[n_q*k], n_pages[n_q]
 * optional final_out[n_q*n] (every final score), z_out[n_q] (Z_b),
 *          shift_out[n_q] (c_b)
 */
static int retrieve_impl(const uint16_t *emb, int64_t n, int32_t dim, const uint16_t *q,
                         int32_t n_q, const int64_t *row_ptr, const int32_t *col, const double *w,
                         double tau, double alpha, int32_t hops, int32_t k,
                         const int32_t *page_of, const int32_t *ns_of, const int32_t *q_ns,
                         const uint8_t *dead, int32_t sort_by_time, int64_t *ids, double *scores,
                         int32_t *page_ids, int32_t *n_pages, double *final_out, double *z_out,
                         double *shift_out);

int ora_retrieve(const uint16_t *emb, int64_t n, int32_t dim, const uint16_t *q, int32_t n_q,
                 const int64_t *row_ptr, const int32_t *col, const double *w, double tau,
                 double alpha, int32_t hops, int32_t k, const int32_t *page_of, int64_t *ids,
                 double *scores, int32_t *page_ids, int32_t *n_pages, double *final_out,
                 double *z_out, double *shift_out)
{
    return retrieve_impl(emb, n, dim, q, n_q, row_ptr, col, w, tau, alpha, hops, k, page_of,
                         NULL, NULL, NULL, 0, ids, scores, page_ids, n_pages, final_out, z_out,
                         shift_out);
}

/*
 * As ora_retrieve, with query b selecting only among the chunks whose
 * ns_of[i] equals q_ns[b] (ns_of[n], q_ns[n_q]; both NULL: no scope), and
 * none of the chunks with dead[i] != 0 (dead[n] or NULL), padded with ID -1
 * when fewer than k remain, and with sort_by_time != 0 returning the
 * selected IDs in ascending ID order.
 */
int ora_retrieve_scoped(const uint16_t *emb, int64_t n, int32_t dim, const uint16_t *q,
                        int32_t n_q, const int64_t *row_ptr, const int32_t *col, const double *w,
                        double tau, double alpha, int32_t hops, int32_t k,
                        const int32_t *page_of, const int32_t *ns_of, const int32_t *q_ns,
                        const uint8_t *dead, int32_t sort_by_time, int64_t *ids, double *scores,
                        int32_t *page_ids, int32_t *n_pages, double *final_out)
{
    if ((ns_of == NULL) != (q_ns == NULL))
        return ORA_EINVAL;
    return retrieve_impl(emb, n, dim, q, n_q, row_ptr, col, w, tau, alpha, hops, k, page_of,
                         ns_of, q_ns, dead, sort_by_time, ids, scores, page_ids, n_pages,
                         final_out, NULL, NULL);
}

/*
 * Deletion of chunks from the relation graph: the CSR without every edge
 * i -> j where dead[i] or dead[j].  new_row_ptr[n+1]; new_col / new_aff with
 * room for nnz entries.  (The weights are then ora_row_softmax of the new
 * logits.)
 */
int ora_drop_dead(int64_t n, const int64_t *row_ptr, const int32_t *col, const float *aff,
                  const uint8_t *dead, int64_t *new_row_ptr, int32_t *new_col, float *new_aff)
{
    if (n < 0 || !row_ptr || !dead || !new_row_ptr)
        return ORA_EINVAL;
    int64_t o = 0;
    new_row_ptr[0] = 0;
    for (int64_t i = 0; i < n; ++i) {
        for (int64_t e = row_ptr[i]; e < row_ptr[i + 1]; ++e) {
            if (dead[i] || dead[col[e]])
                continue;
            new_col[o] = col[e];
            new_aff[o] = aff[e];
            ++o;
        }
        new_row_ptr[i + 1] = o;
    }
    return ORA_OK;
}

/* selected entries of one query by ascending ID (padding -1 stays last) */
static int cmp_id_time(const void *pa, const void *pb)
{
    const ora_pair *a = (const ora_pair *)pa, *b = (const ora_pair *)pb;
    return (a->id < b->id) ? -1 : (a->id > b->id);
}

static int retrieve_impl(const uint16_t *emb, int64_t n, int32_t dim, const uint16_t *q,
                         int32_t n_q, const int64_t *row_ptr, const int32_t *col, const double *w,
                         double tau, double alpha, int32_t hops, int32_t k,
                         const int32_t *page_of, const int32_t *ns_of, const int32_t *q_ns,
                         const uint8_t *dead, int32_t sort_by_time, int64_t *ids, double *scores,
                         int32_t *page_ids, int32_t *n_pages, double *final_out, double *z_out,
                         double *shift_out)
{
    if (n < 1 || dim < 1 || n_q < 0 || k < 1 || k > n || hops < 0 || alpha < 0.0)
        return ORA_EINVAL;
    if (hops > 0 && alpha != 0.0 && (!row_ptr || !col || !w))
        return ORA_EINVAL;
    double *z = (double *)malloc(sizeof(double) * n);
    double *u = (double *)malloc(sizeof(double) * n);
    double *s = (double *)malloc(sizeof(double) * n);
    double *t = (double *)malloc(sizeof(double) * n);
    double *qv = (double *)malloc(sizeof(double) * dim);
    ora_pair *order = (ora_pair *)malloc(sizeof(ora_pair) * n);
    int64_t *pg = (int64_t *)malloc(sizeof(int64_t) * k);
    if (!z || !u || !s || !t || !qv || !order || !pg) {
        free(z); free(u); free(s); free(t); free(qv); free(order); free(pg);
        return ORA_ENOMEM;
    }
    for (int32_t b = 0; b < n_q; ++b) {
        for (int32_t c = 0; c < dim; ++c)
            qv[c] = bf16_widen(q[(int64_t)b * dim + c]);
        /* score */
        double cmax = -INFINITY;
        for (int64_t i = 0; i < n; ++i) {
            const uint16_t *e = emb + i * (int64_t)dim;
            double acc = 0.0;
            for (int32_t c = 0; c < dim; ++c)
                acc += qv[c] * bf16_widen(e[c]);
            z[i] = tau * acc;
            if (z[i] > cmax)
                cmax = z[i];
        }
        double zsum = 0.0;
        for (int64_t i = 0; i < n; ++i) {
            u[i] = (dead && dead[i]) ? 0.0 : exp(z[i] - cmax);   /* deleted: no score */
            zsum += u[i];
        }
        /* propagate: scatter over out-edges */
        for (int64_t i = 0; i < n; ++i)
            s[i] = u[i];
        for (int32_t h = 0; h < hops && alpha != 0.0; ++h) {
            for (int64_t j = 0; j < n; ++j)
                t[j] = 0.0;
            for (int64_t i = 0; i < n; ++i)
                for (int64_t e = row_ptr[i]; e < row_ptr[i + 1]; ++e)
                    t[col[e]] += w[e] * s[i];
            for (int64_t j = 0; j < n; ++j)
                s[j] = u[j] + alpha * t[j];
        }
        int64_t n_cand = 0;
        for (int64_t i = 0; i < n; ++i) {
            s[i] /= zsum;
            if (ns_of && ns_of[i] != q_ns[b])
                continue;   /* outside the query's namespace: not a candidate */
            if (dead && dead[i])
                continue;   /* deleted: not a candidate */
            order[n_cand].key = s[i];
            order[n_cand].id = i;
            ++n_cand;
        }
        if (final_out)
            memcpy(final_out + (int64_t)b * n, s, sizeof(double) * n);
        if (z_out)
            z_out[b] = zsum;
        if (shift_out)
            shift_out[b] = cmax;
        /* top-k by full sort of the candidates */
        qsort(order, (size_t)n_cand, sizeof(ora_pair), cmp_desc_id);
        const int32_t got = n_cand < k ? (int32_t)n_cand : k;
        if (sort_by_time)
            qsort(order, (size_t)got, sizeof(ora_pair), cmp_id_time);
        for (int32_t r = 0; r < k; ++r) {
            ids[(int64_t)b * k + r] = r < got ? order[r].id : -1;
            scores[(int64_t)b * k + r] = r < got ? order[r].key : 0.0;
        }
        /* page resolve */
        if (page_of) {
            for (int32_t r = 0; r < k; ++r) {
                int32_t p = r < got ? page_of[order[r].id] : -1;
                page_ids[(int64_t)b * k + r] = p;
                if (r < got)
                    pg[r] = p;
            }
            qsort(pg, (size_t)got, sizeof(int64_t), cmp_i64);
            int32_t distinct = 0;
            for (int32_t r = 0; r < got; ++r)
                if (r == 0 || pg[r] != pg[r - 1])
                    ++distinct;
            n_pages[b] = distinct;
        }
    }
    free(z); free(u); free(s); free(t); free(qv); free(order); free(pg);
    return ORA_OK;
}

/* ------------------------------------------------------------ relation update */

typedef struct {
    int64_t col;
    float aff;
} ora_edge;

static int cmp_edge_col(const void *pa, const void *pb)
{
    const ora_edge *a = (const ora_edge *)pa, *b = (const ora_edge *)pb;
    return (a->col < b->col) ? -1 : (a->col > b->col);
}

/*
 * emb        (first + n_new) x dim bf16 bits (prior chunks, then the new ones)
 * old CSR    n_rows = first + n_new rows: row_ptr[n_rows+1], col, aff
 *            (rows first .. first+n_new-1 must be empty)
 * new CSR    new_row_ptr[n_rows+1], new_col / new_aff with room for
 *            nnz + n_new*M*(reciprocal ? 2 : 1) entries
 * optional   nbr_ids[n_new*M], nbr_cos[n_new*M]: the selected neighbours in
 *            (cos desc, id asc) order
 */
int ora_update_relations(const uint16_t *emb, int32_t dim, int64_t first, int64_t n_new, int32_t m,
                         double scale, int32_t reciprocal, const int64_t *row_ptr,
                         const int32_t *col, const float *aff, int64_t *new_row_ptr,
                         int32_t *new_col, float *new_aff, int64_t *nbr_ids, double *nbr_cos)
{
    if (dim < 1 || first < 1 || n_new < 0 || m < 1 || m > first)
        return ORA_EINVAL;
    const int64_t n_rows = first + n_new;
    for (int64_t r = first; r < n_rows; ++r)
        if (row_ptr[r + 1] != row_ptr[r])
            return ORA_EINVAL;
    int64_t *sel = (int64_t *)malloc(sizeof(int64_t) * (n_new * m + 1));
    double *selc = (double *)malloc(sizeof(double) * (n_new * m + 1));
    ora_pair *cand = (ora_pair *)malloc(sizeof(ora_pair) * first);
    double *nv = (double *)malloc(sizeof(double) * dim);
    int64_t *extra = (int64_t *)calloc((size_t)n_rows, sizeof(int64_t));
    if (!sel || !selc || !cand || !nv || !extra) {
        free(sel); free(selc); free(cand); free(nv); free(extra);
        return ORA_ENOMEM;
    }
    /* top-M prior neighbours of every new chunk */
    for (int64_t a = 0; a < n_new; ++a) {
        const int64_t nid = first + a;
        for (int32_t c = 0; c < dim; ++c)
            nv[c] = bf16_widen(emb[nid * dim + c]);
        for (int64_t i = 0; i < first; ++i) {
            const uint16_t *e = emb + i * (int64_t)dim;
            double acc = 0.0;
            for (int32_t c = 0; c < dim; ++c)
                acc += nv[c] * bf16_widen(e[c]);
            cand[i].key = acc;
            cand[i].id = i;
        }
        qsort(cand, (size_t)first, sizeof(ora_pair), cmp_desc_id);
        for (int32_t r = 0; r < m; ++r) {
            sel[a * m + r] = cand[r].id;
            selc[a * m + r] = cand[r].key;
            if (nbr_ids)
                nbr_ids[a * m + r] = cand[r].id;
            if (nbr_cos)
                nbr_cos[a * m + r] = cand[r].key;
            extra[nid] += 1;
            if (reciprocal)
                extra[cand[r].id] += 1;
        }
    }
    /* rebuild rows: old edges plus inserted ones, sorted by column */
    int64_t max_row = 0;
    for (int64_t r = 0; r < n_rows; ++r) {
        int64_t len = row_ptr[r + 1] - row_ptr[r] + extra[r];
        if (len > max_row)
            max_row = len;
    }
    ora_edge **rows = (ora_edge **)calloc((size_t)n_rows, sizeof(ora_edge *));
    int64_t *fill = (int64_t *)calloc((size_t)n_rows, sizeof(int64_t));
    int rc = ORA_OK;
    if (!rows || !fill) {
        rc = ORA_ENOMEM;
        goto done;
    }
    for (int64_t r = 0; r < n_rows; ++r) {
        int64_t len = row_ptr[r + 1] - row_ptr[r] + extra[r];
        rows[r] = (ora_edge *)malloc(sizeof(ora_edge) * (size_t)(len > 0 ? len : 1));
        if (!rows[r]) {
            rc = ORA_ENOMEM;
            goto done;
        }
        for (int64_t e = row_ptr[r]; e < row_ptr[r + 1]; ++e) {
            rows[r][fill[r]].col = col[e];
            rows[r][fill[r]].aff = aff[e];
            fill[r] += 1;
        }
    }
    for (int64_t a = 0; a < n_new; ++a) {
        const int64_t nid = first + a;
        for (int32_t r = 0; r < m; ++r) {
            const int64_t j = sel[a * m + r];
            const float lg = (float)(scale * selc[a * m + r]);
            rows[nid][fill[nid]].col = j;
            rows[nid][fill[nid]].aff = lg;
            fill[nid] += 1;
            if (reciprocal) {
                rows[j][fill[j]].col = nid;
                rows[j][fill[j]].aff = lg;
                fill[j] += 1;
            }
        }
    }
    new_row_ptr[0] = 0;
    for (int64_t r = 0; r < n_rows; ++r) {
        qsort(rows[r], (size_t)fill[r], sizeof(ora_edge), cmp_edge_col);
        for (int64_t e = 1; e < fill[r]; ++e)
            if (rows[r][e].col == rows[r][e - 1].col) {
                rc = ORA_EINVAL; /* an edge to that chunk already existed */
                goto done;
            }
        int64_t base = new_row_ptr[r];
        for (int64_t e = 0; e < fill[r]; ++e) {
            new_col[base + e] = (int32_t)rows[r][e].col;
            new_aff[base + e] = rows[r][e].aff;
        }
        new_row_ptr[r + 1] = base + fill[r];
    }
done:
    if (rows)
        for (int64_t r = 0; r < n_rows; ++r)
            free(rows[r]);
    free(rows); free(fill);
    free(sel); free(selc); free(cand); free(nv); free(extra);
    (void)max_row;
    return rc;
}
