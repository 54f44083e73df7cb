// The C ABI declared in include/akashic_mem.h: store lifecycle, appends,
// relation-graph maintenance, retrieval orchestration, read-back, status and
// phase timing.  All arithmetic runs in the kernels of the other files.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <mutex>
#include <string>
#include <unordered_map>
#include <vector>

#include "ak_common.cuh"
#include "ak_update.cuh"

using namespace ak;

// ------------------------------------------------------------------ errors
static thread_local std::string g_last_error;

void ak::set_last_error(const char *msg) { g_last_error = msg ? msg : ""; }

static akashic_status_t fail(akashic_status_t st, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return st;
}

#define CUDA_TRY(call)                                                                         \
    do {                                                                                       \
        cudaError_t e_ = (call);                                                               \
        if (e_ != cudaSuccess)                                                                 \
            return fail(e_ == cudaErrorMemoryAllocation ? AKASHIC_ENOMEM : AKASHIC_ECUDA,      \
                        "%s: %s (%s:%d)", #call, cudaGetErrorString(e_), __FILE__, __LINE__);  \
    } while (0)

#define AK_TRY(call)                                                                           \
    do {                                                                                       \
        akashic_status_t s_ = (call);                                                          \
        if (s_ != AKASHIC_OK) return s_;                                                       \
    } while (0)

// ------------------------------------------------------------------ device buffers
struct DevBuf {
    void *p = nullptr;
    size_t cap = 0;
    ~DevBuf() {
        if (p) cudaFree(p);
    }
    // Grow to at least `bytes`; contents are not preserved unless keep.
    akashic_status_t ensure(size_t bytes, bool keep = false, cudaStream_t st = 0) {
        if (bytes <= cap) return AKASHIC_OK;
        size_t want = bytes < 256 ? 256 : bytes;
        void *q = nullptr;
        cudaError_t e = cudaMalloc(&q, want);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(AKASHIC_ENOMEM, "device allocation of %zu bytes failed", want);
        }
        if (keep && p && cap) {
            e = cudaMemcpyAsync(q, p, cap, cudaMemcpyDeviceToDevice, st);
            if (e == cudaSuccess) e = cudaStreamSynchronize(st);
            if (e != cudaSuccess) {
                cudaFree(q);
                return fail(AKASHIC_ECUDA, "buffer growth copy: %s", cudaGetErrorString(e));
            }
        }
        if (p) cudaFree(p);
        p = q;
        cap = want;
        return AKASHIC_OK;
    }
    template <typename T> T *as() const { return (T *)p; }
};

struct StreamScratch {
    DevBuf qp, shift, u, sa, sb, zpart, partial, cand, counters;
    DevBuf samp, ext_s, zsamp;   // retrieval without hops: the score's row sample
    DevBuf qns, ns_s, dead_s;    // scope: per query column, per sample row
    DevBuf rmax_u, rmin_u;       // u's row maxima / minima over the real queries
    DevBuf ub, lb, ext, pfloor;  // the last hop's row bounds, extremes, floor
    DevBuf skip_split, skip_slot, kept_rows, kept_count, kept_segs, kflag, kpos, ktmp;
    DevBuf reach_keep, reach_part, reach_plan;   // flags + bad + done, partials, plan
    DevBuf nsf;                  // scoped last hop: tags, their floors, their count
    // every candidate's combined coefficients (bf16 hi, lo), and their key
    DevBuf coef_hi, coef_lo;
    uint64_t coef_build = ~0ull;
    float coef_alpha = -1.f;
    int coef_H = 0;
    int64_t coef_n = -1;
    // the call's plan read back: pinned host words and the event after
    // their copy (the host waits for that point only)
    int32_t *plan_host = nullptr;
    cudaEvent_t plan_ev = nullptr;
    ~StreamScratch() {
        if (plan_host) cudaFreeHost(plan_host);
        if (plan_ev) cudaEventDestroy(plan_ev);
    }
};

struct ProfRec {
    int phase;
    cudaEvent_t a, b;
    int launches;
};

struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) cudaSetDevice(dev);
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

struct akashic_mem {
    int device = 0;
    int dim = 0;
    int64_t cap = 0;
    int per_page = 1;
    float tau = 0.f;
    float rel_scale = 10.f;
    int64_t n = 0;
    int64_t next_page = 0;
    // chunks live in HBM in page order: row r holds chunk ext_of[r], chunk c
    // is in row row_of[c]; page_of is indexed by row
    DevBuf emb, page_of, ext_of, row_of, max_norm, status;
    DevBuf ns_row;               // namespace tag of the chunk in each row (0 by default)
    DevBuf dead_row;             // 1 in the rows of deleted chunks
    bool has_dead = false;       // any chunk deleted (enables the masks)
    // memory manager: per-page slot counters, co-retrieval statistics
    DevBuf page_total, page_live, sel, co_key, co_val, mm_ctr;
    int64_t page_cap = 0, co_cap = 0, co_upper = 0;
    int64_t appended = 0, moves = 0;
    // canonical out-edge CSR
    int64_t nnz = 0;
    DevBuf row_ptr, col, aff, w;
    // in-edge transpose + split plan for the propagation hop
    DevBuf in_ptr, in_src, in_w, in_aff;
    DevBuf rstat;                // per chunk ID: (max, 1/sum) of its out-row softmax
    // spares the relation update writes the next CSR / transpose into (then
    // swapped with the live arrays), and grow-only scratch for its temporaries
    DevBuf rp2, col2, aff2, in_ptr2, in_src2, in_aff2, in_w2;
    DevBuf scr[SCR_COUNT];
    bool inc_transpose = true;   // relation updates patch the transpose instead of re-sorting
    SplitParams split;
    bool fuse_filter = true;     // top-k filter in the last hop's epilogue
    bool hop_prune = true;       // last hop skips rows bounded below every filter threshold
    int64_t n_split = 0, n_segs = 0;
    DevBuf split_row, split_slot0, seg_e0, seg_e1, seg_slot, split_order, slot_split;
    // graph-only mass vectors of the last hop's row bounds, levels 0..mass_levels
    // (recomputed lazily after the graph changes)
    DevBuf mass_up, mass_dn, mass_zero, mass_vu, mass_vl;
    int mass_levels = -1;
    int64_t mass_n = -1;      // rows they were computed for
    // reach coefficients of the candidate rows (ak_reach.cu), same lifetime
    DevBuf reach_rows, reach_t, reach_map, reach_c;
    int reach_levels = -1;
    int reach_T = 0;          // candidate rows (host copy)
    int64_t reach_n = -1;     // rows they were computed for
    uint64_t reach_build = 0; // incremented by every rebuild
    bool reach_on = true;     // AKASHIC_REACH=0: always run the hops
    // the mass levels and reach tables are built by whichever retrieve needs
    // them first, on its own stream: table_mu serialises the builders and
    // every retrieve that reads them waits on table_ev, recorded after the
    // last build (retrieves on other streams may run concurrently)
    std::mutex table_mu;
    cudaEvent_t table_ev = nullptr;
    std::mutex mu;
    std::unordered_map<void *, StreamScratch *> scratch;
    // profiling
    bool prof = false;
    std::vector<ProfRec> recs;
    std::vector<cudaEvent_t> ev_pool;
    ~akashic_mem() {
        for (auto &kv : scratch) delete kv.second;
        for (auto &r : recs) {
            cudaEventDestroy(r.a);
            cudaEventDestroy(r.b);
        }
        for (auto e : ev_pool) cudaEventDestroy(e);
        if (table_ev) cudaEventDestroy(table_ev);
    }
};

// ------------------------------------------------------------------ profiling helpers
struct PhaseScope {
    akashic_mem *m;
    int phase;
    cudaStream_t st;
    cudaEvent_t a = nullptr;
    int launches = 0;
    PhaseScope(akashic_mem *m_, int ph, cudaStream_t s) : m(m_), phase(ph), st(s) {
        if (!m->prof) return;
        a = take_event();
        if (a) cudaEventRecord(a, st);
    }
    cudaEvent_t take_event() {
        std::lock_guard<std::mutex> g(m->mu);
        cudaEvent_t e = nullptr;
        if (!m->ev_pool.empty()) {
            e = m->ev_pool.back();
            m->ev_pool.pop_back();
        } else if (cudaEventCreate(&e) != cudaSuccess) {
            cudaGetLastError();
            e = nullptr;
        }
        return e;
    }
    // close the scope early (once); the destructor then does nothing
    void end() {
        if (!m->prof || !a) return;
        cudaEvent_t b = take_event();
        if (b) {
            cudaEventRecord(b, st);
            std::lock_guard<std::mutex> g(m->mu);
            m->recs.push_back(ProfRec{phase, a, b, launches});
        }
        a = nullptr;
    }
    ~PhaseScope() {
        if (!m->prof || !a) return;
        cudaEvent_t b = take_event();
        if (!b) return;
        cudaEventRecord(b, st);
        std::lock_guard<std::mutex> g(m->mu);
        m->recs.push_back(ProfRec{phase, a, b, launches});
    }
};

// ------------------------------------------------------------------ small kernels
__global__ void k_page_max(const int32_t *page_of, int64_t n, int *out_max, int *status) {
    int best = -1;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        int p = page_of[i];
        if (p < 0) set_status(status, AKASHIC_EDEVICE);
        best = p > best ? p : best;
    }
    atomicMax(out_max, best);
}

// row_ptr of the appended rows in the store's CSR: dst[r] = base + src[r] - src[0]
__global__ void k_rebase_ptr(const int64_t *src, int64_t *dst, int64_t n1, int64_t base) {
    const int64_t p0 = src ? src[0] : 0;
    for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n1;
         r += (int64_t)gridDim.x * blockDim.x)
        dst[r] = src ? base + src[r] - p0 : base;
}

static int bits_for(int64_t max_value) {
    int b = 0;
    while (b < 32 && ((int64_t)1 << b) <= max_value) ++b;
    return b;
}

static akashic_status_t check_status(akashic_mem *m, cudaStream_t st, const char *what) {
    CUDA_TRY(cudaStreamSynchronize(st));
    int code = 0;
    CUDA_TRY(cudaMemcpy(&code, m->status.p, sizeof(int), cudaMemcpyDeviceToHost));
    if (code != 0) {
        CUDA_TRY(cudaMemset(m->status.p, 0, sizeof(int)));
        return fail((akashic_status_t)code, "%s: device reported status %d", what, code);
    }
    return AKASHIC_OK;
}

// Grow-only scratch of a store (UpdateArgs::scratch): 1/8 headroom when a
// slot has to grow, so slowly growing sizes do not reallocate every call.
static void *store_scratch(void *ctx, int slot, size_t bytes) {
    akashic_mem *m = (akashic_mem *)ctx;
    if (slot < 0 || slot >= SCR_COUNT) return nullptr;
    DevBuf &b = m->scr[slot];
    if (bytes > b.cap && b.ensure(bytes + bytes / 8) != AKASHIC_OK) return nullptr;
    return b.p;
}

static MmTables mm_tables(akashic_mem *m) {
    MmTables t;
    t.page_total = m->page_total.as<int32_t>();
    t.page_live = m->page_live.as<int32_t>();
    t.sel = m->sel.as<int32_t>();
    t.co_key = m->co_key.as<unsigned long long>();
    t.co_val = m->co_val.as<uint32_t>();
    t.co_cap = m->co_cap;
    t.next_page = m->mm_ctr.as<int64_t>();
    t.writes = m->mm_ctr.as<int64_t>() + 1;
    t.released = m->mm_ctr.as<unsigned long long>() + 2;
    return t;
}

// Page counters for page IDs below `need` (grown by doubling, new tail zeroed).
static akashic_status_t mm_ensure_pages(akashic_mem *m, int64_t need, cudaStream_t st) {
    if (need <= m->page_cap) return AKASHIC_OK;
    int64_t cap = m->page_cap > 0 ? m->page_cap : 1024;
    while (cap < need) cap *= 2;
    AK_TRY(m->page_total.ensure((size_t)cap * 4, true, st));
    AK_TRY(m->page_live.ensure((size_t)cap * 4, true, st));
    CUDA_TRY(cudaMemsetAsync(m->page_total.as<int32_t>() + m->page_cap, 0,
                             (size_t)(cap - m->page_cap) * 4, st));
    CUDA_TRY(cudaMemsetAsync(m->page_live.as<int32_t>() + m->page_cap, 0,
                             (size_t)(cap - m->page_cap) * 4, st));
    m->page_cap = cap;
    return AKASHIC_OK;
}

// Co-retrieval table able to take `more` new pairs at load <= 1/2.
static akashic_status_t mm_ensure_pairs(akashic_mem *m, int64_t more, cudaStream_t st,
                                        int *launches = nullptr) {
    if (m->co_cap > 0 && m->co_upper + more <= m->co_cap / 2) return AKASHIC_OK;
    int64_t cap = m->co_cap > 0 ? m->co_cap : ((int64_t)1 << 20);
    while (m->co_upper + more > cap / 2) cap *= 2;
    DevBuf nk, nv;
    AK_TRY(nk.ensure((size_t)cap * 8));
    AK_TRY(nv.ensure((size_t)cap * 4));
    std::swap(m->co_key.p, nk.p);
    std::swap(m->co_key.cap, nk.cap);
    std::swap(m->co_val.p, nv.p);
    std::swap(m->co_val.cap, nv.cap);
    const int64_t old_cap = m->co_cap;
    m->co_cap = cap;
    CUDA_TRY(launch_mm_rehash(nk.as<unsigned long long>(), nv.as<uint32_t>(), old_cap,
                              mm_tables(m), m->status.as<int>(), st));
    if (launches && old_cap > 0) *launches += 1;
    CUDA_TRY(cudaStreamSynchronize(st));   // the old table is freed on return
    return AKASHIC_OK;
}

// A scratch buffer seen through the DevBuf-like accessors.
struct Tmp {
    void *p;
    size_t cap;
    template <typename T> T *as() const { return (T *)p; }
};

// Grow a spare buffer with 1/4 headroom (contents not kept).
static akashic_status_t ensure_spare(DevBuf &b, size_t bytes) {
    return bytes > b.cap ? b.ensure(bytes + bytes / 4) : AKASHIC_OK;
}

static akashic_status_t build_split_plan(akashic_mem *m, cudaStream_t st);

// Rebuild the in-edge transpose (stable by source, hence sorted by source
// within each destination), its weights, and the split plan of long rows.
static akashic_status_t rebuild_in_edges(akashic_mem *m, cudaStream_t st) {
    const int64_t n = m->n, nnz = m->nnz;
    AK_TRY(m->in_ptr.ensure((size_t)(m->cap + 1) * sizeof(int64_t)));
    AK_TRY(m->in_src.ensure((size_t)(nnz > 0 ? nnz : 1) * sizeof(int32_t)));
    AK_TRY(m->in_w.ensure((size_t)(nnz > 0 ? nnz : 1) * sizeof(float)));
    AK_TRY(m->in_aff.ensure((size_t)(nnz > 0 ? nnz : 1) * sizeof(float)));
    DevBuf src, keys, vals, keys2, vals2, tmp, deg;
    const size_t tmp_bytes = (radix_tmp_bytes(nnz) > scan_tmp_bytes(n + 1) ? radix_tmp_bytes(nnz)
                                                                             : scan_tmp_bytes(n + 1)) +
                             4096;
    AK_TRY(tmp.ensure(tmp_bytes));
    AK_TRY(deg.ensure((size_t)(n + 1) * sizeof(int64_t) * 2));
    if (nnz > 0) {
        AK_TRY(src.ensure((size_t)nnz * 4));
        AK_TRY(keys.ensure((size_t)nnz * 4));
        AK_TRY(vals.ensure((size_t)nnz * 4));
        AK_TRY(keys2.ensure((size_t)nnz * 4));
        AK_TRY(vals2.ensure((size_t)nnz * 4));
        const int32_t *row_of = m->row_of.as<int32_t>();
        CUDA_TRY(launch_edge_src_check(m->row_ptr.as<int64_t>(), m->col.as<int32_t>(), n, 0, n,
                                       src.as<int32_t>(), m->status.as<int>(), st));
        // edges ordered by (target row, source row): sort by source row, then
        // stably by target row
        CUDA_TRY(launch_map_keys(nullptr, src.as<int32_t>(), row_of, keys.as<uint32_t>(), nnz, st));
        CUDA_TRY(launch_iota(vals.as<uint32_t>(), nnz, st));
        bool alt = false;
        CUDA_TRY(radix_sort_pairs(keys.as<uint32_t>(), vals.as<uint32_t>(), keys2.as<uint32_t>(),
                                  vals2.as<uint32_t>(), nnz, bits_for(n - 1), tmp.p, tmp.cap, st,
                                  &alt));
        uint32_t *k1 = alt ? keys2.as<uint32_t>() : keys.as<uint32_t>();
        uint32_t *v1 = alt ? vals2.as<uint32_t>() : vals.as<uint32_t>();
        uint32_t *k2 = alt ? keys.as<uint32_t>() : keys2.as<uint32_t>();
        uint32_t *v2 = alt ? vals.as<uint32_t>() : vals2.as<uint32_t>();
        CUDA_TRY(launch_map_keys(v1, m->col.as<int32_t>(), row_of, k1, nnz, st));
        bool alt2 = false;
        CUDA_TRY(radix_sort_pairs(k1, v1, k2, v2, nnz, bits_for(n - 1), tmp.p, tmp.cap, st, &alt2));
        const uint32_t *order = alt2 ? v2 : v1;
        CUDA_TRY(launch_gather_in(order, src.as<int32_t>(), row_of, m->w.as<float>(),
                                  m->aff.as<float>(), m->in_src.as<int32_t>(), m->in_w.as<float>(),
                                  m->in_aff.as<float>(), nnz, st));
    }
    int64_t *degp = deg.as<int64_t>();
    CUDA_TRY(cudaMemsetAsync(degp, 0, (size_t)(n + 1) * sizeof(int64_t), st));
    CUDA_TRY(launch_in_degree(m->col.as<int32_t>(), m->row_of.as<int32_t>(), nnz, degp, st));
    CUDA_TRY(scan_exclusive(degp, m->in_ptr.as<int64_t>(), n, tmp.p, tmp.cap, st));
    return build_split_plan(m, st);
}

// Split plan: hub rows cut into window segments, segments in window-major
// order, split rows heaviest first.
static akashic_status_t build_split_plan(akashic_mem *m, cudaStream_t st) {
    const int64_t n = m->n;
    m->mass_levels = -1;   // the graph changed
    m->reach_levels = -1;
    // temporaries from the store's scratch (slots SCR_SPLIT0..11)
    akashic_status_t sc_rc = AKASHIC_OK;
    auto get = [&](int i, size_t bytes) -> Tmp {
        void *q = store_scratch(m, SCR_SPLIT0 + i, bytes);
        if (!q) sc_rc = AKASHIC_ENOMEM;
        return Tmp{q, bytes};
    };
    const Tmp tmp = get(0, scan_tmp_bytes(n + 1) + 4096);
    const Tmp nseg = get(1, (size_t)(n + 1) * 8), flag = get(2, (size_t)(n + 1) * 8);
    const Tmp slot_off = get(3, (size_t)(n + 1) * 8), split_idx = get(4, (size_t)(n + 1) * 8);
    if (sc_rc != AKASHIC_OK) return fail(sc_rc, "relation graph rebuild: out of device memory");
    CUDA_TRY(launch_split_count(m->split, m->in_ptr.as<int64_t>(), m->in_src.as<int32_t>(), n,
                                nseg.as<int64_t>(), flag.as<int64_t>(), st));
    CUDA_TRY(scan_exclusive(nseg.as<int64_t>(), slot_off.as<int64_t>(), n, tmp.p, tmp.cap, st));
    CUDA_TRY(scan_exclusive(flag.as<int64_t>(), split_idx.as<int64_t>(), n, tmp.p, tmp.cap, st));
    int64_t n_segs = 0, n_split = 0;
    CUDA_TRY(cudaMemcpyAsync(&n_segs, slot_off.as<int64_t>() + n, 8, cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaMemcpyAsync(&n_split, split_idx.as<int64_t>() + n, 8, cudaMemcpyDeviceToHost, st));
    AK_TRY(check_status(m, st, "relation graph rebuild"));
    if (n_segs > 0x7fffffffLL) return fail(AKASHIC_ECAPACITY, "too many hub segments");
    m->n_segs = n_segs;
    m->n_split = n_split;
    if (n_split > 0) {
        // grown with headroom: every relation update adds a few segments, and
        // a reallocation would synchronise the device
        AK_TRY(ensure_spare(m->split_row, (size_t)n_split * 4));
        AK_TRY(ensure_spare(m->split_slot0, (size_t)(n_split + 1) * 8));
        AK_TRY(ensure_spare(m->seg_e0, (size_t)n_segs * 8));
        AK_TRY(ensure_spare(m->seg_e1, (size_t)n_segs * 8));
        AK_TRY(ensure_spare(m->seg_slot, (size_t)n_segs * 4));
        const Tmp e0 = get(5, (size_t)n_segs * 8), e1 = get(6, (size_t)n_segs * 8);
        const Tmp win = get(7, (size_t)n_segs * 4), order = get(8, (size_t)n_segs * 4);
        const Tmp win2 = get(9, (size_t)n_segs * 4), order2 = get(10, (size_t)n_segs * 4);
        const Tmp rtmp = get(11, radix_tmp_bytes(n_segs) + 4096);
        if (sc_rc != AKASHIC_OK) return fail(sc_rc, "relation graph rebuild: out of device memory");
        CUDA_TRY(launch_split_fill(m->split, m->in_ptr.as<int64_t>(), m->in_src.as<int32_t>(), n,
                                   nseg.as<int64_t>(), slot_off.as<int64_t>(),
                                   split_idx.as<int64_t>(), m->split_row.as<int32_t>(),
                                   m->split_slot0.as<int64_t>(), e0.as<int64_t>(),
                                   e1.as<int64_t>(), win.as<uint32_t>(), st));
        CUDA_TRY(cudaMemcpyAsync(m->split_slot0.as<int64_t>() + n_split, &n_segs, 8,
                                 cudaMemcpyHostToDevice, st));
        CUDA_TRY(launch_iota(order.as<uint32_t>(), n_segs, st));
        bool alt = false;
        CUDA_TRY(radix_sort_pairs(win.as<uint32_t>(), order.as<uint32_t>(), win2.as<uint32_t>(),
                                  order2.as<uint32_t>(), n_segs, bits_for((n - 1) / m->split.win_rows),
                                  rtmp.p, rtmp.cap, st, &alt));
        CUDA_TRY(launch_seg_permute(alt ? order2.as<uint32_t>() : order.as<uint32_t>(),
                                    e0.as<int64_t>(), e1.as<int64_t>(), n_segs,
                                    m->seg_e0.as<int64_t>(), m->seg_e1.as<int64_t>(),
                                    m->seg_slot.as<int32_t>(), st));
        // split rows heaviest first (the hop's fixup order)
        AK_TRY(ensure_spare(m->split_order, (size_t)n_split * 4));
        CUDA_TRY(launch_split_keys(m->split_slot0.as<int64_t>(), n_split, win.as<uint32_t>(),
                                   order.as<uint32_t>(), st));
        bool alt2 = false;
        CUDA_TRY(radix_sort_pairs(win.as<uint32_t>(), order.as<uint32_t>(), win2.as<uint32_t>(),
                                  order2.as<uint32_t>(), n_split, 32, rtmp.p, rtmp.cap, st, &alt2));
        CUDA_TRY(cudaMemcpyAsync(m->split_order.p, alt2 ? order2.p : order.p, (size_t)n_split * 4,
                                 cudaMemcpyDeviceToDevice, st));
        AK_TRY(ensure_spare(m->slot_split, (size_t)n_segs * 4));
        CUDA_TRY(launch_slot_owner(m->split_slot0.as<int64_t>(), n_split,
                                   m->slot_split.as<int32_t>(), st));
        AK_TRY(check_status(m, st, "relation graph rebuild"));
    }
    return check_status(m, st, "relation graph rebuild");
}

// ================================================================== ABI
extern "C" {

const char *akashic_mem_last_error(void) { return g_last_error.c_str(); }

akashic_status_t akashic_mem_create(const akashic_mem_config_t *cfg, akashic_mem_t **out) {
    g_last_error.clear();
    if (!cfg || !out) return fail(AKASHIC_EINVAL, "create: NULL argument");
    *out = nullptr;
    if (cfg->dim < 64 || cfg->dim > 4096 || cfg->dim % 64 != 0)
        return fail(AKASHIC_EINVAL, "create: dim must be a multiple of 64 in [64, 4096]");
    if (cfg->capacity < 1 || cfg->capacity > 0x7fffffffLL)
        return fail(AKASHIC_EINVAL, "create: capacity must be in [1, 2^31-1]");
    if (cfg->chunks_per_page < 1) return fail(AKASHIC_EINVAL, "create: chunks_per_page < 1");
    if (!(cfg->temperature >= 0.f) || !isfinite(cfg->temperature) ||
        !(cfg->relation_scale >= 0.f) || !isfinite(cfg->relation_scale))
        return fail(AKASHIC_EINVAL, "create: temperature/relation_scale must be finite and >= 0");
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || cfg->device < 0 || cfg->device >= ndev) {
        cudaGetLastError();
        return fail(AKASHIC_EINVAL, "create: no CUDA device %d", cfg->device);
    }
    DeviceGuard g(cfg->device);
    akashic_mem *m = new (std::nothrow) akashic_mem();
    if (!m) return fail(AKASHIC_ENOMEM, "create: host allocation failed");
    m->device = cfg->device;
    m->dim = cfg->dim;
    m->cap = cfg->capacity;
    m->per_page = cfg->chunks_per_page;
    m->tau = cfg->temperature > 0.f ? cfg->temperature : 1.0f / sqrtf((float)cfg->dim);
    m->rel_scale = cfg->relation_scale > 0.f ? cfg->relation_scale : 10.f;
    // propagation plan knobs (tuning only; results do not depend on them
    // beyond fp32 summation order)
    if (const char *v = getenv("AKASHIC_SPLIT_T")) m->split.split_t = atoll(v) > 0 ? atoll(v) : m->split.split_t;
    if (const char *v = getenv("AKASHIC_SEG_LEN")) m->split.seg_len = atoll(v) > 0 ? atoll(v) : m->split.seg_len;
    if (const char *v = getenv("AKASHIC_FUSE_FILTER")) m->fuse_filter = atoi(v) != 0;
    if (const char *v = getenv("AKASHIC_HOP_PRUNE")) m->hop_prune = atoi(v) != 0;
    if (const char *v = getenv("AKASHIC_REACH")) m->reach_on = atoi(v) != 0;
    if (const char *v = getenv("AKASHIC_FULL_TRANSPOSE")) m->inc_transpose = atoi(v) == 0;
    if (const char *v = getenv("AKASHIC_WIN_ROWS")) m->split.win_rows = atoll(v) > 0 ? atoll(v) : m->split.win_rows;
    akashic_status_t s;
    if ((s = m->emb.ensure((size_t)m->cap * m->dim * 2)) != AKASHIC_OK ||
        (s = m->page_of.ensure((size_t)m->cap * 4)) != AKASHIC_OK ||
        (s = m->ext_of.ensure((size_t)m->cap * 4)) != AKASHIC_OK ||
        (s = m->row_of.ensure((size_t)m->cap * 4)) != AKASHIC_OK ||
        (s = m->max_norm.ensure(4)) != AKASHIC_OK || (s = m->status.ensure(4)) != AKASHIC_OK ||
        (s = m->rstat.ensure((size_t)m->cap * 8)) != AKASHIC_OK ||
        (s = m->ns_row.ensure((size_t)m->cap * 4)) != AKASHIC_OK ||
        (s = m->dead_row.ensure((size_t)m->cap * 4)) != AKASHIC_OK ||
        (s = m->row_ptr.ensure((size_t)(m->cap + 1) * 8)) != AKASHIC_OK ||
        (s = m->in_ptr.ensure((size_t)(m->cap + 1) * 8)) != AKASHIC_OK) {
        delete m;
        return s;
    }
    if (cudaMemset(m->max_norm.p, 0, 4) != cudaSuccess || cudaMemset(m->status.p, 0, 4) != cudaSuccess ||
        cudaMemset(m->row_ptr.p, 0, 8) != cudaSuccess || cudaMemset(m->in_ptr.p, 0, 8) != cudaSuccess ||
        cudaMemset(m->ns_row.p, 0, (size_t)m->cap * 4) != cudaSuccess ||
        cudaMemset(m->dead_row.p, 0, (size_t)m->cap * 4) != cudaSuccess ||
        m->sel.ensure((size_t)m->cap * 4) != AKASHIC_OK ||
        cudaMemset(m->sel.p, 0, (size_t)m->cap * 4) != cudaSuccess ||
        m->mm_ctr.ensure(32) != AKASHIC_OK || cudaMemset(m->mm_ctr.p, 0, 32) != cudaSuccess ||
        mm_ensure_pages(m, 1024, 0) != AKASHIC_OK || mm_ensure_pairs(m, 0, 0) != AKASHIC_OK ||
        cudaDeviceSynchronize() != cudaSuccess) {
        delete m;
        return fail(AKASHIC_ECUDA, "create: initialisation failed");
    }
    *out = m;
    return AKASHIC_OK;
}

void akashic_mem_destroy(akashic_mem_t *m) {
    if (!m) return;
    DeviceGuard g(m->device);
    cudaDeviceSynchronize();
    delete m;
}

akashic_status_t akashic_mem_size(const akashic_mem_t *m, int64_t *n_chunks, int64_t *nnz) {
    if (!m) return fail(AKASHIC_EINVAL, "size: NULL store");
    if (n_chunks) *n_chunks = m->n;
    if (nnz) *nnz = m->nnz;
    return AKASHIC_OK;
}

akashic_status_t akashic_mem_sync(akashic_mem_t *m, void *stream) {
    if (!m) return fail(AKASHIC_EINVAL, "sync: NULL store");
    DeviceGuard g(m->device);
    return check_status(m, (cudaStream_t)stream, "sync");
}

akashic_status_t akashic_mem_check_wait_timeout(akashic_mem_t *m, uint32_t polls, void *stream) {
    g_last_error.clear();
    if (!m) return fail(AKASHIC_EINVAL, "check_wait_timeout: NULL store");
    if (polls < 1 || polls > (1u << 26))
        return fail(AKASHIC_EINVAL, "check_wait_timeout: polls must be in [1, 2^26]");
    DeviceGuard g(m->device);
    CUDA_TRY(launch_wait_timeout_check(m->status.as<int>(), polls, (cudaStream_t)stream));
    return AKASHIC_OK;
}

akashic_status_t akashic_mem_sort_pairs(uint32_t *keys, uint32_t *vals, int64_t n, int32_t bits,
                                        void *stream) {
    g_last_error.clear();
    if (n < 0 || n > 0x7fffffffLL || bits < 0 || bits > 32 || (n > 1 && (!keys || !vals)))
        return fail(AKASHIC_EINVAL, "sort_pairs: bad n, bits or buffers");
    if (n <= 1 || bits == 0) return AKASHIC_OK;
    cudaStream_t st = (cudaStream_t)stream;
    const size_t words = ((size_t)n * 8 + 255) & ~(size_t)255;
    const size_t tb = radix_tmp_bytes(n) + 4096;
    void *buf = nullptr;
    if (cudaMalloc(&buf, words + tb) != cudaSuccess) {
        cudaGetLastError();
        return fail(AKASHIC_ENOMEM, "sort_pairs: %lld bytes of scratch", (long long)(words + tb));
    }
    uint32_t *k2 = (uint32_t *)buf, *v2 = k2 + n;
    bool alt = false;
    cudaError_t e = radix_sort_pairs(keys, vals, k2, v2, n, bits, (uint8_t *)buf + words, tb, st,
                                     &alt);
    if (e == cudaSuccess && alt)
        e = cudaMemcpyAsync(keys, k2, (size_t)n * 4, cudaMemcpyDeviceToDevice, st);
    if (e == cudaSuccess && alt)
        e = cudaMemcpyAsync(vals, v2, (size_t)n * 4, cudaMemcpyDeviceToDevice, st);
    const cudaError_t es = cudaStreamSynchronize(st);
    if (e == cudaSuccess) e = es;
    cudaFree(buf);
    if (e != cudaSuccess) return fail(AKASHIC_ECUDA, "sort_pairs: %s", cudaGetErrorString(e));
    return AKASHIC_OK;
}

akashic_status_t akashic_mem_append_chunks(akashic_mem_t *m, const uint16_t *emb, int64_t n,
                                           const int32_t *page_of, const int64_t *row_ptr,
                                           const int32_t *col, const float *aff,
                                           int64_t *first_id_out, void *stream) {
    g_last_error.clear();
    if (!m) return fail(AKASHIC_EINVAL, "append: NULL store");
    if (n < 0 || (n > 0 && !emb)) return fail(AKASHIC_EINVAL, "append: bad n or emb");
    if (((uintptr_t)emb & 15u) != 0) return fail(AKASHIC_EINVAL, "append: emb must be 16-byte aligned");
    const bool has_edges = row_ptr != nullptr;
    if (!row_ptr && (col || aff))
        return fail(AKASHIC_EINVAL, "append: col/aff given without row_ptr");
    if (m->n + n > m->cap)
        return fail(AKASHIC_ECAPACITY, "append: %lld + %lld chunks exceed capacity %lld",
                    (long long)m->n, (long long)n, (long long)m->cap);
    if (first_id_out) *first_id_out = m->n;
    if (n == 0) return AKASHIC_OK;
    DeviceGuard g(m->device);
    cudaStream_t st = (cudaStream_t)stream;
    const int64_t first = m->n;
    PhaseScope ph(m, AKASHIC_PHASE_GRAPH, st);
    // -- validate the new edges before anything is committed
    int64_t e_lo = 0, e_hi = 0;
    if (has_edges) {
        CUDA_TRY(cudaMemcpyAsync(&e_lo, row_ptr, 8, cudaMemcpyDeviceToHost, st));
        CUDA_TRY(cudaMemcpyAsync(&e_hi, row_ptr + n, 8, cudaMemcpyDeviceToHost, st));
        CUDA_TRY(launch_edge_src_check(row_ptr, col, n, first, first + n, nullptr,
                                       m->status.as<int>(), st));
        AK_TRY(check_status(m, st, "append: edge check"));
        if (e_hi < e_lo) return fail(AKASHIC_EINVAL, "append: row_ptr decreases");
        if (m->has_dead && e_hi > e_lo && col) {
            CUDA_TRY(launch_check_dead_targets(col + e_lo, e_hi - e_lo, first,
                                               m->row_of.as<int32_t>(), m->dead_row.as<int32_t>(),
                                               m->status.as<int>(), st));
            AK_TRY(check_status(m, st, "append: an edge points at a deleted chunk"));
        }
        if (e_hi > e_lo && !(col && aff))
            return fail(AKASHIC_EINVAL, "append: edges given without col or aff");
        if (m->nnz + (e_hi - e_lo) > 0x7fffffffLL)
            return fail(AKASHIC_ECAPACITY, "append: more than 2^31-1 relation edges");
    }
    int64_t max_page = -1;
    if (page_of) {
        DevBuf pm;
        AK_TRY(pm.ensure(4));
        int init = -1;
        CUDA_TRY(cudaMemcpyAsync(pm.p, &init, 4, cudaMemcpyHostToDevice, st));
        k_page_max<<<device_sm_count(), 256, 0, st>>>(page_of, n, pm.as<int>(), m->status.as<int>());
        CUDA_TRY(cudaGetLastError());
        int mx = -1;
        CUDA_TRY(cudaMemcpyAsync(&mx, pm.p, 4, cudaMemcpyDeviceToHost, st));
        AK_TRY(check_status(m, st, "append: page_of must be >= 0"));
        max_page = mx;
    }
    const int64_t new_nnz = e_hi - e_lo;
    if (new_nnz > 0) {
        const size_t need = (size_t)(m->nnz + new_nnz);
        size_t grow = need + need / 4;
        AK_TRY(m->col.ensure(grow * 4, true, st));
        AK_TRY(m->aff.ensure(grow * 4, true, st));
        AK_TRY(m->w.ensure(grow * 4, true, st));
    }
    // -- the batch's rows in page order (stable: ID order within a page)
    DevBuf okeys, ovals, okeys2, ovals2, otmp;
    const uint32_t *order = nullptr;
    if (page_of && max_page > 0 && n > 1) {
        AK_TRY(okeys.ensure((size_t)n * 4));
        AK_TRY(ovals.ensure((size_t)n * 4));
        AK_TRY(okeys2.ensure((size_t)n * 4));
        AK_TRY(ovals2.ensure((size_t)n * 4));
        AK_TRY(otmp.ensure(radix_tmp_bytes(n) + 4096));
        CUDA_TRY(cudaMemcpyAsync(okeys.p, page_of, (size_t)n * 4, cudaMemcpyDeviceToDevice, st));
        CUDA_TRY(launch_iota(ovals.as<uint32_t>(), n, st));
        bool alt = false;
        CUDA_TRY(radix_sort_pairs(okeys.as<uint32_t>(), ovals.as<uint32_t>(), okeys2.as<uint32_t>(),
                                  ovals2.as<uint32_t>(), n, bits_for(max_page), otmp.p, otmp.cap,
                                  st, &alt));
        order = alt ? ovals2.as<uint32_t>() : ovals.as<uint32_t>();
    }
    // -- commit
    CUDA_TRY(launch_batch_layout(order, first, n, m->dim, emb, m->emb.as<uint16_t>(), page_of,
                                 m->next_page, m->per_page, m->page_of.as<int32_t>(),
                                 m->ext_of.as<int32_t>(), m->row_of.as<int32_t>(), st));
    if (page_of) {
        if (max_page + 1 > m->next_page) m->next_page = max_page + 1;
    } else {
        m->next_page += ceil_div<int64_t>(n, m->per_page);
    }
    // the new chunks occupy a slot of their pages
    AK_TRY(mm_ensure_pages(m, m->next_page + 1, st));
    CUDA_TRY(launch_mm_count_pages(m->page_of.as<int32_t>(), first, n, mm_tables(m), st));
    m->appended += n;
    CUDA_TRY(launch_row_norm_max(m->emb.as<uint16_t>() + first * m->dim, n, m->dim,
                                 m->max_norm.as<float>(), st));
    int64_t *rp = m->row_ptr.as<int64_t>() + first;   // rp[0] is already m->nnz
    k_rebase_ptr<<<device_sm_count() * 4, 256, 0, st>>>(has_edges ? row_ptr : nullptr, rp, n + 1,
                                                         m->nnz);
    CUDA_TRY(cudaGetLastError());
    if (new_nnz > 0) {
        CUDA_TRY(cudaMemcpyAsync(m->col.as<int32_t>() + m->nnz, col + e_lo, (size_t)new_nnz * 4,
                                 cudaMemcpyDeviceToDevice, st));
        CUDA_TRY(cudaMemcpyAsync(m->aff.as<float>() + m->nnz, aff + e_lo, (size_t)new_nnz * 4,
                                 cudaMemcpyDeviceToDevice, st));
        CUDA_TRY(launch_row_softmax(rp, m->aff.as<float>(), m->w.as<float>(), n,
                                    m->rstat.as<float2>() + first, st));
    }
    m->n += n;
    m->nnz += new_nnz;
    if (new_nnz == 0 && first > 0) {
        // no new edges: the new rows have no in-edges, the transpose and the
        // hub plan are unchanged; only the row pointers are extended
        k_rebase_ptr<<<device_sm_count() * 4, 256, 0, st>>>(nullptr, m->in_ptr.as<int64_t>() + first + 1,
                                                             n, m->nnz);
        CUDA_TRY(cudaGetLastError());
        return check_status(m, st, "append");
    }
    AK_TRY(rebuild_in_edges(m, st));
    return AKASHIC_OK;
}

akashic_status_t akashic_mem_update_relations(akashic_mem_t *m, int64_t first, int64_t n,
                                              int32_t M, int32_t reciprocal, void *stream) {
    g_last_error.clear();
    if (!m) return fail(AKASHIC_EINVAL, "update: NULL store");
    if (first < 0 || n < 0 || first + n > m->n)
        return fail(AKASHIC_EINVAL, "update: range [%lld, %lld) outside the store of %lld",
                    (long long)first, (long long)(first + n), (long long)m->n);
    if (M < 1 || M > 64 || M > first)
        return fail(AKASHIC_EINVAL, "update: M must be in [1, min(64, first)]");
    if (n == 0) return AKASHIC_OK;
    DeviceGuard g(m->device);
    cudaStream_t st = (cudaStream_t)stream;
    // rows [first, first+n) must have no out-edges
    int64_t a = 0, b = 0;
    CUDA_TRY(cudaMemcpyAsync(&a, m->row_ptr.as<int64_t>() + first, 8, cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaMemcpyAsync(&b, m->row_ptr.as<int64_t>() + first + n, 8, cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaStreamSynchronize(st));
    if (a != b) return fail(AKASHIC_EINVAL, "update: rows [first, first+n) already have out-edges");
    UpdateArgs ua;
    ua.emb = m->emb.as<uint16_t>();
    ua.dim = m->dim;
    ua.n_rows = m->n;
    ua.first = first;
    ua.n_new = n;
    ua.M = M;
    ua.reciprocal = reciprocal != 0;
    ua.scale = m->rel_scale;
    ua.status = m->status.as<int>();
    ua.ext_of = m->ext_of.as<int32_t>();
    ua.row_of = m->row_of.as<int32_t>();
    int64_t nnz_new = m->nnz + n * M * (reciprocal ? 2 : 1);
    if (nnz_new > 0x7fffffffLL)
        return fail(AKASHIC_ECAPACITY, "update: more than 2^31-1 relation edges");
    ua.scratch = store_scratch;
    ua.scratch_ctx = m;
    ua.dead_row = m->has_dead ? m->dead_row.as<int32_t>() : nullptr;
    ua.nbr_ids = (int32_t *)store_scratch(m, SCR_NBR_IDS, (size_t)n * M * 4);
    ua.nbr_cos = (float *)store_scratch(m, SCR_NBR_COS, (size_t)n * M * 4);
    if (!ua.nbr_ids || !ua.nbr_cos) return fail(AKASHIC_ENOMEM, "update: out of device memory");
    DevBuf &ncol = m->col2, &naff = m->aff2, &nrp = m->rp2;
    AK_TRY(ensure_spare(ncol, (size_t)nnz_new * 4));
    AK_TRY(ensure_spare(naff, (size_t)nnz_new * 4));
    AK_TRY(ensure_spare(nrp, (size_t)(m->cap + 1) * 8));
    {
        PhaseScope ph(m, AKASHIC_PHASE_RELATE, st);
        akashic_status_t r = relate_top_m(ua, st, &ph.launches);
        if (r != AKASHIC_OK) return fail(r, "update: relation GEMM / top-M failed");
        AK_TRY(check_status(m, st, "update: top-M"));
    }
    {
        PhaseScope ph(m, AKASHIC_PHASE_GRAPH, st);
        {
            PhaseScope pc(m, AKASHIC_PHASE_CSR_INSERT, st);
            akashic_status_t r = csr_insert(ua, m->row_ptr.as<int64_t>(), m->col.as<int32_t>(),
                                            m->aff.as<float>(), m->nnz, nrp.as<int64_t>(),
                                            ncol.as<int32_t>(), naff.as<float>(), st,
                                            &pc.launches);
            ph.launches += pc.launches;
            if (r != AKASHIC_OK) return fail(r, "update: CSR insert failed");
            AK_TRY(check_status(m, st, "update"));
        }
        PhaseScope pt(m, AKASHIC_PHASE_TRANSPOSE, st);
        std::swap(m->row_ptr.p, nrp.p);
        std::swap(m->row_ptr.cap, nrp.cap);
        std::swap(m->col.p, ncol.p);
        std::swap(m->col.cap, ncol.cap);
        std::swap(m->aff.p, naff.p);
        std::swap(m->aff.cap, naff.cap);
        const int64_t nnz_old = m->nnz;
        m->nnz = nnz_new;
        AK_TRY(m->w.ensure(m->col.cap, false));
        CUDA_TRY(launch_row_softmax(m->row_ptr.as<int64_t>(), m->aff.as<float>(), m->w.as<float>(),
                                    m->n, m->rstat.as<float2>(), st));
        pt.launches += 1;
        if (!m->inc_transpose || nnz_old == 0) {
            AK_TRY(rebuild_in_edges(m, st));
        } else {
            // patch the transpose: old lists moved, new edges placed, weights
            // recomputed from the logits (ak_inedges.cu)
            DevBuf &ptr2 = m->in_ptr2, &src2 = m->in_src2, &aff2 = m->in_aff2, &w2 = m->in_w2;
            const int64_t rows = m->n, pairs = n * (int64_t)M;
            AK_TRY(ensure_spare(ptr2, (size_t)(m->cap + 1) * 8));
            AK_TRY(ensure_spare(src2, (size_t)nnz_new * 4));
            AK_TRY(ensure_spare(aff2, (size_t)nnz_new * 4));
            AK_TRY(ensure_spare(w2, (size_t)nnz_new * 4));
            const size_t tb = (radix_tmp_bytes(pairs) > scan_tmp_bytes(rows + 1)
                                   ? radix_tmp_bytes(pairs) : scan_tmp_bytes(rows + 1)) + 4096;
            void *p_inc = store_scratch(m, SCR_IN_INC, (size_t)(rows + 1) * 8);
            void *p_deg = store_scratch(m, SCR_IN_DEG, (size_t)(rows + 1) * 8);
            void *p_off = store_scratch(m, SCR_IN_OFF, (size_t)(rows + 1) * 8);
            void *p_rs = store_scratch(m, SCR_IN_RSTAT, (size_t)(rows > 0 ? rows : 1) * 8);
            void *p_k = store_scratch(m, SCR_KEYS, (size_t)pairs * 4 + 16);
            void *p_v = store_scratch(m, SCR_VALS, (size_t)pairs * 4 + 16);
            void *p_k2 = store_scratch(m, SCR_KEYS2, (size_t)pairs * 4 + 16);
            void *p_v2 = store_scratch(m, SCR_VALS2, (size_t)pairs * 4 + 16);
            void *p_tmp = store_scratch(m, SCR_TMP, tb);
            if (!p_inc || !p_deg || !p_off || !p_rs || !p_k || !p_v || !p_k2 || !p_v2 || !p_tmp)
                return fail(AKASHIC_ENOMEM, "update: out of device memory");
            InEdgeUpdate u;
            u.n = rows;
            u.nnz_new = nnz_new;
            u.in_ptr_old = m->in_ptr.as<int64_t>();
            u.in_src_old = m->in_src.as<int32_t>();
            u.in_aff_old = m->in_aff.as<float>();
            u.in_ptr_new = ptr2.as<int64_t>();
            u.in_src_new = src2.as<int32_t>();
            u.in_aff_new = aff2.as<float>();
            u.in_w_new = w2.as<float>();
            u.nbr_ids = ua.nbr_ids;
            u.nbr_cos = ua.nbr_cos;
            u.scale = m->rel_scale;
            u.first = first;
            u.n_new = n;
            u.M = M;
            u.reciprocal = reciprocal != 0;
            u.row_bits = bits_for(rows - 1);
            u.row_of = m->row_of.as<int32_t>();
            u.ext_of = m->ext_of.as<int32_t>();
            u.rstat = m->rstat.as<float2>();
            InEdgeScratch sc{(int64_t *)p_inc, (int64_t *)p_deg, (int64_t *)p_off,
                             (uint32_t *)p_k, (uint32_t *)p_v, (uint32_t *)p_k2, (uint32_t *)p_v2,
                             p_tmp, tb, (float2 *)p_rs};
            CUDA_TRY(launch_in_edges_update(u, sc, st, &pt.launches));
            std::swap(m->in_ptr.p, ptr2.p);
            std::swap(m->in_ptr.cap, ptr2.cap);
            std::swap(m->in_src.p, src2.p);
            std::swap(m->in_src.cap, src2.cap);
            std::swap(m->in_aff.p, aff2.p);
            std::swap(m->in_aff.cap, aff2.cap);
            std::swap(m->in_w.p, w2.p);
            std::swap(m->in_w.cap, w2.cap);
            pt.end();
            ph.launches += pt.launches;
            PhaseScope phub(m, AKASHIC_PHASE_HUB_PLAN, st);
            AK_TRY(build_split_plan(m, st));
        }
    }
    return AKASHIC_OK;
}

static StreamScratch *scratch_for(akashic_mem *m, void *stream) {
    std::lock_guard<std::mutex> g(m->mu);
    auto it = m->scratch.find(stream);
    if (it != m->scratch.end()) return it->second;
    StreamScratch *s = new (std::nothrow) StreamScratch();
    if (s) m->scratch[stream] = s;
    return s;
}

static akashic_status_t retrieve_impl(akashic_mem *m, const uint16_t *q, int32_t B, int32_t k,
                                      float alpha, int32_t hops, const int32_t *q_ns,
                                      int32_t sort_by_time, int64_t *ids, float *scores,
                                      int32_t *page_ids, int32_t *n_pages, void *stream);

akashic_status_t akashic_mem_retrieve(akashic_mem_t *m, const uint16_t *q, int32_t B, int32_t k,
                                      float alpha, int32_t hops, int64_t *ids, float *scores,
                                      int32_t *page_ids, int32_t *n_pages, void *stream) {
    g_last_error.clear();
    return retrieve_impl(m, q, B, k, alpha, hops, nullptr, 0, ids, scores, page_ids, n_pages,
                         stream);
}

akashic_status_t akashic_mem_retrieve_scoped(akashic_mem_t *m, const uint16_t *q, int32_t B,
                                             int32_t k, float alpha, int32_t hops,
                                             const int32_t *q_ns, int32_t sort_by_time,
                                             int64_t *ids, float *scores, int32_t *page_ids,
                                             int32_t *n_pages, void *stream) {
    g_last_error.clear();
    return retrieve_impl(m, q, B, k, alpha, hops, q_ns, sort_by_time, ids, scores, page_ids,
                         n_pages, stream);
}

akashic_status_t akashic_mem_set_namespace(akashic_mem_t *m, int64_t first, int64_t n,
                                           const int32_t *ns, void *stream) {
    g_last_error.clear();
    if (!m) return fail(AKASHIC_EINVAL, "set_namespace: NULL store");
    if (first < 0 || n < 0 || first + n > m->n)
        return fail(AKASHIC_EINVAL, "set_namespace: range [%lld, %lld) outside the store of %lld",
                    (long long)first, (long long)(first + n), (long long)m->n);
    if (n == 0) return AKASHIC_OK;
    if (!ns) return fail(AKASHIC_EINVAL, "set_namespace: NULL ns");
    DeviceGuard g(m->device);
    CUDA_TRY(launch_scatter_by_row(ns, m->row_of.as<int32_t>(), first, n, m->ns_row.as<int32_t>(),
                                   (cudaStream_t)stream));
    return AKASHIC_OK;
}
akashic_status_t akashic_mem_delete(akashic_mem_t *m, const int64_t *ids, int64_t n,
                                    void *stream) {
    g_last_error.clear();
    if (!m) return fail(AKASHIC_EINVAL, "delete: NULL store");
    if (n < 0) return fail(AKASHIC_EINVAL, "delete: n < 0");
    if (n == 0) return AKASHIC_OK;
    if (!ids) return fail(AKASHIC_EINVAL, "delete: NULL ids");
    DeviceGuard g(m->device);
    cudaStream_t st = (cudaStream_t)stream;
    // check every ID first, so that a bad list changes nothing
    CUDA_TRY(launch_mark_dead(ids, n, m->n, m->row_of.as<int32_t>(), nullptr,
                              m->status.as<int>(), st));
    AK_TRY(check_status(m, st, "delete: chunk IDs must lie in [0, size)"));
    CUDA_TRY(launch_mark_dead(ids, n, m->n, m->row_of.as<int32_t>(), m->dead_row.as<int32_t>(),
                              m->status.as<int>(), st, m->page_of.as<int32_t>(),
                              m->page_live.as<int32_t>()));
    m->has_dead = true;
    const int64_t rows = m->n, nnz = m->nnz;
    if (nnz == 0) return AKASHIC_OK;
    const size_t tb = scan_tmp_bytes(nnz + 1) + 4096;
    int64_t *keep = (int64_t *)store_scratch(m, SCR_DEL_KEEP, (size_t)(nnz + 1) * 8);
    int64_t *pos = (int64_t *)store_scratch(m, SCR_DEL_POS, (size_t)(nnz + 1) * 8);
    void *tmp = store_scratch(m, SCR_DEL_TMP, tb);
    if (!keep || !pos || !tmp) return fail(AKASHIC_ENOMEM, "delete: out of device memory");
    // out-edge CSR (rows are chunk IDs, targets chunk IDs)
    AK_TRY(ensure_spare(m->rp2, (size_t)(m->cap + 1) * 8));
    AK_TRY(ensure_spare(m->col2, (size_t)nnz * 4));
    AK_TRY(ensure_spare(m->aff2, (size_t)nnz * 4));
    DropDead d{rows, nnz, m->row_ptr.as<int64_t>(), m->col.as<int32_t>(), m->aff.as<float>(),
               m->row_of.as<int32_t>(), m->dead_row.as<int32_t>(), ids, n, rows, nullptr,
               keep, pos, tmp, tb, m->rp2.as<int64_t>(), m->col2.as<int32_t>(),
               m->aff2.as<float>()};
    CUDA_TRY(launch_drop_dead_edges(d, st));
    int64_t nnz_new = 0;
    CUDA_TRY(cudaMemcpyAsync(&nnz_new, pos + nnz, 8, cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaStreamSynchronize(st));
    std::swap(m->row_ptr.p, m->rp2.p);
    std::swap(m->row_ptr.cap, m->rp2.cap);
    std::swap(m->col.p, m->col2.p);
    std::swap(m->col.cap, m->col2.cap);
    std::swap(m->aff.p, m->aff2.p);
    std::swap(m->aff.cap, m->aff2.cap);
    m->nnz = nnz_new;
    AK_TRY(m->w.ensure(m->col.cap > 4 ? m->col.cap : 4, false));
    CUDA_TRY(launch_row_softmax(m->row_ptr.as<int64_t>(), m->aff.as<float>(), m->w.as<float>(),
                                rows, m->rstat.as<float2>(), st));
    // in-edge transpose (rows are store rows, sources rows); the same edges go
    AK_TRY(ensure_spare(m->in_ptr2, (size_t)(m->cap + 1) * 8));
    AK_TRY(ensure_spare(m->in_src2, (size_t)nnz * 4));
    AK_TRY(ensure_spare(m->in_aff2, (size_t)nnz * 4));
    AK_TRY(ensure_spare(m->in_w2, (size_t)nnz * 4));
    DropDead di{rows, nnz, m->in_ptr.as<int64_t>(), m->in_src.as<int32_t>(), m->in_aff.as<float>(),
                nullptr, m->dead_row.as<int32_t>(), ids, n, rows, m->row_of.as<int32_t>(),
                keep, pos, tmp, tb, m->in_ptr2.as<int64_t>(), m->in_src2.as<int32_t>(),
                m->in_aff2.as<float>()};
    CUDA_TRY(launch_drop_dead_edges(di, st));
    CUDA_TRY(launch_in_weights(m->in_src2.as<int32_t>(), m->in_aff2.as<float>(), nnz_new,
                               m->ext_of.as<int32_t>(), m->rstat.as<float2>(),
                               m->in_w2.as<float>(), st));
    std::swap(m->in_ptr.p, m->in_ptr2.p);
    std::swap(m->in_ptr.cap, m->in_ptr2.cap);
    std::swap(m->in_src.p, m->in_src2.p);
    std::swap(m->in_src.cap, m->in_src2.cap);
    std::swap(m->in_aff.p, m->in_aff2.p);
    std::swap(m->in_aff.cap, m->in_aff2.cap);
    std::swap(m->in_w.p, m->in_w2.p);
    std::swap(m->in_w.cap, m->in_w2.cap);
    AK_TRY(build_split_plan(m, st));
    return check_status(m, st, "delete");
}
akashic_status_t akashic_mem_relocate(akashic_mem_t *m, const int64_t *S, int32_t n_req,
                                      int32_t s_len, float tau_assoc, void *stream) {
    g_last_error.clear();
    if (!m) return fail(AKASHIC_EINVAL, "relocate: NULL store");
    if (n_req < 0 || s_len < 1 || s_len > 64)
        return fail(AKASHIC_EINVAL, "relocate: need n_req >= 0 and 1 <= s_len <= 64");
    if (!(tau_assoc >= 0.f && tau_assoc <= 1.f))
        return fail(AKASHIC_EINVAL, "relocate: tau_assoc must lie in [0, 1]");
    if (n_req == 0) return AKASHIC_OK;
    if (!S) return fail(AKASHIC_EINVAL, "relocate: NULL S");
    DeviceGuard g(m->device);
    cudaStream_t st = (cudaStream_t)stream;
    PhaseScope ph(m, AKASHIC_PHASE_RELOCATE, st);
    const int64_t pairs = (int64_t)n_req * s_len * (s_len - 1) / 2;
    AK_TRY(mm_ensure_pairs(m, pairs, st, &ph.launches));
    AK_TRY(mm_ensure_pages(m, m->next_page + (int64_t)n_req * ceil_div<int64_t>(64, m->per_page) + 1,
                           st));
    int32_t *gb = (int32_t *)store_scratch(m, SCR_MM_G, (size_t)n_req * 64 * 4);
    int32_t *gn = (int32_t *)store_scratch(m, SCR_MM_GN, (size_t)n_req * 4);
    if (!gb || !gn) return fail(AKASHIC_ENOMEM, "relocate: out of device memory");
    int64_t ctr[2] = {m->next_page, 0};
    CUDA_TRY(cudaMemcpyAsync(m->mm_ctr.p, ctr, 16, cudaMemcpyHostToDevice, st));
    const int32_t *dead = m->has_dead ? m->dead_row.as<int32_t>() : nullptr;
    const MmTables t = mm_tables(m);
    CUDA_TRY(launch_mm_count(S, n_req, s_len, m->n, m->row_of.as<int32_t>(), dead, t,
                             m->status.as<int>(), st));
    CUDA_TRY(launch_mm_relocate(S, n_req, s_len, m->n, m->row_of.as<int32_t>(), dead,
                                m->page_of.as<int32_t>(), t, tau_assoc, m->per_page, gb, gn, st));
    ph.launches += 3;
    CUDA_TRY(cudaMemcpyAsync(ctr, m->mm_ctr.p, 16, cudaMemcpyDeviceToHost, st));
    AK_TRY(check_status(m, st, "relocate"));
    m->next_page = ctr[0];
    m->moves += ctr[1];
    m->co_upper += pairs;
    return AKASHIC_OK;
}

akashic_status_t akashic_mem_compact_pages(akashic_mem_t *m, float theta, float tau_assoc,
                                           int64_t *released, void *stream) {
    g_last_error.clear();
    if (!m) return fail(AKASHIC_EINVAL, "compact: NULL store");
    if (!(theta > 0.f && theta <= 1.f))
        return fail(AKASHIC_EINVAL, "compact: theta must lie in (0, 1]");
    if (!(tau_assoc >= 0.f && tau_assoc <= 1.f))
        return fail(AKASHIC_EINVAL, "compact: tau_assoc must lie in [0, 1]");
    DeviceGuard g(m->device);
    cudaStream_t st = (cudaStream_t)stream;
    const int64_t n = m->n, pages = m->next_page;
    if (released) *released = 0;
    if (n == 0) return AKASHIC_OK;
    const size_t tb = (scan_tmp_bytes(n + 1) > radix_tmp_bytes(n) ? scan_tmp_bytes(n + 1)
                                                                   : radix_tmp_bytes(n)) + 4096;
    int32_t *cand = (int32_t *)store_scratch(m, SCR_MM_CAND, (size_t)(pages + 1) * 4);
    int64_t *moving = (int64_t *)store_scratch(m, SCR_MM_MOVING, (size_t)(n + 1) * 8);
    int64_t *pos = (int64_t *)store_scratch(m, SCR_MM_POS, (size_t)(n + 1) * 8);
    int32_t *parent = (int32_t *)store_scratch(m, SCR_MM_PARENT, (size_t)n * 4);
    int32_t *ns_id = (int32_t *)store_scratch(m, SCR_MM_NS, (size_t)n * 4);
    uint32_t *ids = (uint32_t *)store_scratch(m, SCR_MM_IDS, (size_t)n * 4 + 16);
    uint32_t *root = (uint32_t *)store_scratch(m, SCR_MM_ROOT, (size_t)n * 4 + 16);
    uint32_t *nsk = (uint32_t *)store_scratch(m, SCR_MM_NSK, (size_t)n * 4 + 16);
    uint32_t *k2 = (uint32_t *)store_scratch(m, SCR_MM_K2, (size_t)n * 4 + 16);
    uint32_t *v2 = (uint32_t *)store_scratch(m, SCR_MM_V2, (size_t)n * 4 + 16);
    void *tmp = store_scratch(m, SCR_MM_TMP, tb);
    if (!cand || !moving || !pos || !parent || !ns_id || !ids || !root || !nsk || !k2 || !v2 || !tmp)
        return fail(AKASHIC_ENOMEM, "compact: out of device memory");
    PhaseScope ph(m, AKASHIC_PHASE_COMPACT, st);
    const MmTables t = mm_tables(m);
    const int32_t *dead = m->has_dead ? m->dead_row.as<int32_t>() : nullptr;
    const int32_t *row_of = m->row_of.as<int32_t>();
    CUDA_TRY(cudaMemsetAsync(t.released, 0, 8, st));
    CUDA_TRY(launch_mm_compact_prepare(t, pages, theta, n, row_of, dead, m->page_of.as<int32_t>(),
                                       cand, moving, parent, st));
    CUDA_TRY(cudaMemsetAsync(moving + n, 0, 8, st));
    CUDA_TRY(launch_by_id(m->ns_row.as<int32_t>(), row_of, n, ns_id, st));
    CUDA_TRY(launch_mm_union(t, moving, ns_id, tau_assoc, parent, m->status.as<int>(), st));
    ph.launches += (pages > 0) + 3;
    CUDA_TRY(scan_exclusive(moving, pos, n + 1, tmp, tb, st, &ph.launches));
    // released pages and moving chunks, read back together
    CUDA_TRY(cudaMemcpyAsync(t.released + 1, pos + n, 8, cudaMemcpyDeviceToDevice, st));
    int64_t rc[2] = {0, 0};
    CUDA_TRY(cudaMemcpyAsync(rc, t.released, 16, cudaMemcpyDeviceToHost, st));
    AK_TRY(check_status(m, st, "compact"));
    const int64_t n_rel = rc[0], count = rc[1];
    if (count > 0) {
        CUDA_TRY(launch_mm_keys(moving, pos, n, parent, ns_id, ids, root, nsk, st));
        // order (namespace, group root, chunk ID): the list is in ID order;
        // stable sorts by root, then by namespace
        bool alt = false;
        CUDA_TRY(radix_sort_pairs(root, ids, k2, v2, count, 32, tmp, tb, st, &alt, &ph.launches));
        uint32_t *sid = alt ? v2 : ids, *spare_v = alt ? ids : v2;
        uint32_t *nk = alt ? root : k2;
        CUDA_TRY(launch_mm_ns_keys(sid, count, ns_id, nsk, st));
        bool alt2 = false;
        CUDA_TRY(radix_sort_pairs(nsk, sid, nk, spare_v, count, 32, tmp, tb, st, &alt2,
                                  &ph.launches));
        const uint32_t *order = alt2 ? spare_v : sid;
        const uint32_t *ns_sorted = alt2 ? nk : nsk;
        // every namespace starts on a fresh page (compaction never mixes
        // tenants or sessions): pages per namespace run, scanned into each
        // run's base page; `moving` and `pos` are free again
        CUDA_TRY(launch_mm_part_pages(ns_sorted, count, m->per_page, moving, st));
        CUDA_TRY(scan_exclusive(moving, pos, count, tmp, tb, st, &ph.launches));
        int64_t new_pages = 0;
        CUDA_TRY(cudaMemcpyAsync(&new_pages, pos + count, 8, cudaMemcpyDeviceToHost, st));
        AK_TRY(check_status(m, st, "compact"));
        AK_TRY(mm_ensure_pages(m, m->next_page + new_pages + 1, st));
        CUDA_TRY(launch_mm_release_repack(mm_tables(m), pages, cand, order, ns_sorted, pos, count,
                                          row_of, m->page_of.as<int32_t>(), m->next_page,
                                          m->per_page, st));
        ph.launches += 3 + (pages > 0) + 1;
        m->next_page += new_pages;
        m->moves += count;
    } else if (n_rel > 0) {
        CUDA_TRY(launch_mm_release_repack(t, pages, cand, nullptr, nullptr, nullptr, 0, row_of,
                                          m->page_of.as<int32_t>(), m->next_page, m->per_page,
                                          st));
        ph.launches += 1;
    }
    if (released) *released = n_rel;
    return check_status(m, st, "compact");
}

akashic_status_t akashic_mem_page_stats(akashic_mem_t *m, int64_t *out) {
    g_last_error.clear();
    if (!m || !out) return fail(AKASHIC_EINVAL, "page_stats: NULL argument");
    DeviceGuard g(m->device);
    unsigned long long *d = (unsigned long long *)store_scratch(m, SCR_MM_TMP, 64);
    if (!d) return fail(AKASHIC_ENOMEM, "page_stats: out of device memory");
    CUDA_TRY(launch_mm_stats(mm_tables(m), m->next_page, d, 0));
    unsigned long long h[3] = {0, 0, 0};
    CUDA_TRY(cudaMemcpy(h, d, sizeof h, cudaMemcpyDeviceToHost));
    out[0] = (int64_t)h[0];
    out[1] = (int64_t)h[1];
    out[2] = (int64_t)h[2];
    out[3] = m->appended + m->moves;
    out[4] = m->appended;
    return AKASHIC_OK;
}

akashic_status_t akashic_mem_export_pages(akashic_mem_t *m, int32_t *page_of, void *stream) {
    g_last_error.clear();
    if (!m || !page_of) return fail(AKASHIC_EINVAL, "export_pages: NULL argument");
    DeviceGuard g(m->device);
    CUDA_TRY(launch_by_id(m->page_of.as<int32_t>(), m->row_of.as<int32_t>(), m->n, page_of,
                          (cudaStream_t)stream));
    return AKASHIC_OK;
}
}  // extern "C"

// Orders `st` after every earlier table build (any stream); called with
// table_mu held, before the tables are read or extended.
static akashic_status_t wait_tables(akashic_mem *m, cudaStream_t st) {
    if (m->table_ev) CUDA_TRY(cudaStreamWaitEvent(st, m->table_ev, 0));
    return AKASHIC_OK;
}

// Records the end of a table build on `st` (table_mu held).
static akashic_status_t tables_built(akashic_mem *m, cudaStream_t st) {
    if (!m->table_ev) CUDA_TRY(cudaEventCreateWithFlags(&m->table_ev, cudaEventDisableTiming));
    CUDA_TRY(cudaEventRecord(m->table_ev, st));
    return AKASHIC_OK;
}

// Mass levels 0..H of the row bounds (level 0 all ones), extended as needed.
// Room for the largest hop count is taken at once, so extending the levels
// never moves a buffer that a retrieve on another stream may be reading.
// table_mu held.
static akashic_status_t ensure_mass(akashic_mem *m, const HopPlan &hp, int H, cudaStream_t st) {
    const int64_t n = m->n;
    AK_TRY(wait_tables(m, st));
    if (m->mass_n != n) m->mass_levels = -1;
    if (m->mass_levels >= H) return AKASHIC_OK;
    const size_t lv = (size_t)(AKASHIC_MAX_HOPS + 1) * n * 4;
    if (m->mass_levels < 0 || m->mass_up.cap < lv) {
        AK_TRY(ensure_spare(m->mass_up, lv));
        AK_TRY(ensure_spare(m->mass_dn, lv));
        AK_TRY(ensure_spare(m->mass_zero, (size_t)n * 4));
        AK_TRY(ensure_spare(m->mass_vu, (size_t)(m->n_split + 1) * 4));
        AK_TRY(ensure_spare(m->mass_vl, (size_t)(m->n_split + 1) * 4));
        CUDA_TRY(cudaMemsetAsync(m->mass_zero.p, 0, (size_t)n * 4, st));
        CUDA_TRY(launch_fill_f32(m->mass_up.as<float>(), n, 1.f, st));
        CUDA_TRY(launch_fill_f32(m->mass_dn.as<float>(), n, 1.f, st));
        m->mass_levels = 0;
        m->mass_n = n;
    }
    CUDA_TRY(launch_mass_levels(hp, m->mass_levels + 1, H, m->mass_up.as<float>(),
                                m->mass_dn.as<float>(), m->mass_zero.as<float>(),
                                m->mass_vu.as<float>(), m->mass_vl.as<float>(), st));
    m->mass_levels = H;
    return tables_built(m, st);
}

// Reach coefficients of the candidate rows for H hops (after the mass
// levels).  table_mu held.
static akashic_status_t ensure_reach(akashic_mem *m, const HopPlan &hp, int H, cudaStream_t st) {
    const int64_t n = m->n;
    AK_TRY(wait_tables(m, st));
    if (m->reach_levels == H && m->reach_n == n) return AKASHIC_OK;
    AK_TRY(m->reach_rows.ensure(REACH_T * 4));
    AK_TRY(m->reach_t.ensure(16));
    AK_TRY(ensure_spare(m->reach_map, (size_t)n * 4));
    AK_TRY(ensure_spare(m->reach_c, (size_t)H * n * REACH_T * 4));
    ReachBuild rb{};
    rb.n = n;
    rb.n_split = m->n_split;
    rb.H = H;
    rb.split_row = hp.split_row;
    rb.split_order = hp.split_order;
    rb.mup = m->mass_up.as<float>();
    rb.in_ptr = hp.in_ptr;
    rb.in_src = hp.in_src;
    rb.in_w = hp.in_w;
    rb.row_ptr = m->row_ptr.as<int64_t>();
    rb.col = m->col.as<int32_t>();
    rb.row_of = m->row_of.as<int32_t>();
    rb.w = m->w.as<float>();
    rb.rows = m->reach_rows.as<int32_t>();
    rb.t_cnt = m->reach_t.as<int>();
    rb.map = m->reach_map.as<int32_t>();
    rb.C = m->reach_c.as<float>();
    CUDA_TRY(launch_reach_build(rb, st));
    int t = 0;
    CUDA_TRY(cudaMemcpyAsync(&t, m->reach_t.p, 4, cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaStreamSynchronize(st));
    m->reach_T = t;
    m->reach_levels = H;
    m->reach_n = n;
    ++m->reach_build;
    return tables_built(m, st);
}

static akashic_status_t retrieve_impl(akashic_mem *m, const uint16_t *q, int32_t B, int32_t k,
                                      float alpha, int32_t hops, const int32_t *q_ns,
                                      int32_t sort_by_time, int64_t *ids, float *scores,
                                      int32_t *page_ids, int32_t *n_pages, void *stream) {
    if (!m) return fail(AKASHIC_EINVAL, "retrieve: NULL store");
    if (!q || !ids || !scores) return fail(AKASHIC_EINVAL, "retrieve: NULL q/ids/scores");
    if (B < 1) return fail(AKASHIC_EINVAL, "retrieve: B < 1");
    if (k < 1 || k > 64) return fail(AKASHIC_EINVAL, "retrieve: k must be in [1, 64]");
    if (k > m->n) return fail(AKASHIC_EINVAL, "retrieve: k=%d exceeds the %lld chunks", k, (long long)m->n);
    if (hops < 0 || hops > AKASHIC_MAX_HOPS) return fail(AKASHIC_EINVAL, "retrieve: hops must be in [0, 16]");
    if (!(alpha >= 0.f) || !isfinite(alpha)) return fail(AKASHIC_EINVAL, "retrieve: alpha must be finite and >= 0");
    DeviceGuard g(m->device);
    cudaStream_t st = (cudaStream_t)stream;
    StreamScratch *sc = scratch_for(m, stream);
    if (!sc) return fail(AKASHIC_ENOMEM, "retrieve: host allocation failed");
    const int64_t n = m->n;
    const int eff_hops = (alpha > 0.f && m->nnz > 0) ? hops : 0;
    const int sms = device_sm_count();
    for (int32_t off = 0; off < B; off += 256) {
        const int b = B - off < 256 ? B - off : 256;
        int bp = 32;
        while (bp < b) bp <<= 1;
        const int64_t tiles = score_tiles(n);
        int zrows = 0;
        const SelectPlan sp = select_plan(n, bp, k, sms);
        AK_TRY(sc->qp.ensure((size_t)bp * m->dim * 2));
        AK_TRY(sc->shift.ensure((size_t)bp * 4));
        AK_TRY(ensure_spare(sc->u, (size_t)n * bp * 4));
        AK_TRY(ensure_spare(sc->zpart, (size_t)tiles * bp * 4));
        AK_TRY(ensure_spare(sc->cand, (size_t)sp.words * 8));
        if (eff_hops >= 1) AK_TRY(ensure_spare(sc->sa, (size_t)n * bp * 4));
        if (eff_hops >= 2) AK_TRY(ensure_spare(sc->sb, (size_t)n * bp * 4));
        if (eff_hops >= 1 && m->n_segs > 0) AK_TRY(ensure_spare(sc->partial, (size_t)m->n_segs * bp * 4));
        if (eff_hops >= 1) AK_TRY(sc->counters.ensure(64));
        // row bounds for the last hop (fused filter only)
        const bool prune = eff_hops >= 1 && m->fuse_filter && m->hop_prune;
        if (prune) {
            AK_TRY(ensure_spare(sc->rmax_u, (size_t)n * 4));
            AK_TRY(ensure_spare(sc->rmin_u, (size_t)n * 4));
            AK_TRY(ensure_spare(sc->ub, (size_t)n * 4));
            AK_TRY(ensure_spare(sc->lb, (size_t)n * 4));
            AK_TRY(sc->ext.ensure(16));
            AK_TRY(ensure_spare(sc->skip_split, (size_t)(m->n_split + 1) * 4));
            AK_TRY(ensure_spare(sc->kept_rows, (size_t)n * 4));
            AK_TRY(sc->kept_count.ensure(16));
            AK_TRY(ensure_spare(sc->kept_segs, (size_t)(m->n_segs + 1) * 4));
            const int64_t nk = n > m->n_segs ? n : m->n_segs;
            AK_TRY(ensure_spare(sc->kflag, (size_t)(nk + 1) * 8));
            AK_TRY(ensure_spare(sc->kpos, (size_t)(nk + 1) * 8));
            AK_TRY(ensure_spare(sc->ktmp, scan_tmp_bytes(nk + 1) + 4096));
            AK_TRY(ensure_spare(sc->skip_slot, (size_t)(m->n_segs + 1) * 4));
            AK_TRY(sc->pfloor.ensure(16));
        }
        const uint16_t *qb = q + (int64_t)off * m->dim;
        // namespace scope of this batch's queries (padding columns get -1)
        NsScope ns{};
        if (q_ns) {
            AK_TRY(sc->qns.ensure((size_t)bp * 4));
            CUDA_TRY(cudaMemsetAsync(sc->qns.p, 0xff, (size_t)bp * 4, st));
            CUDA_TRY(cudaMemcpyAsync(sc->qns.p, q_ns + off, (size_t)b * 4,
                                     cudaMemcpyDeviceToDevice, st));
            ns = NsScope{m->ns_row.as<int32_t>(), sc->qns.as<int32_t>(), nullptr};
        }
        if (m->has_dead) ns.dead = m->dead_row.as<int32_t>();
        // Without hops the top-k filter is fused into the score GEMM, which
        // then writes no slab: the bound comes from the score of every
        // stride-th row, computed first by the same kernel (same values).
        const SelectPlan sp2 = select_plan(sp.n_sample, bp, k, sms, 1);
        const bool dense_fused = eff_hops == 0 && m->fuse_filter && sp2.off_tr == sp.off_tr &&
                                 sp2.words <= sp.words;
        unsigned long long *ws = sc->cand.as<unsigned long long>();
        ColumnRecompute rc{};
        // the two-hop reach path is tried (its plan may still send the call
        // through the hops): the score GEMM then writes u as split bf16, the
        // operand form the candidates' tensor-core pass loads, in the bytes
        // of the fp32 slab (hi [n][bp], then lo [n][bp])
        const bool reach_try = prune && eff_hops == 2 && !q_ns && m->reach_on &&
                               m->n_split > 0 && (bp == 256 || bp == 128);
        uint16_t *u_hi = reach_try ? sc->u.as<uint16_t>() : nullptr;
        uint16_t *u_lo = reach_try ? u_hi + (size_t)n * bp : nullptr;
        auto score_fp32 = [&](int *launches) -> cudaError_t {
            return launch_score(m->emb.as<uint16_t>(), n, m->dim, sc->qp.as<uint16_t>(), bp,
                                sc->shift.as<float>(), m->tau, sc->u.as<float>(),
                                sc->zpart.as<float>(), m->status.as<int>(), st, launches, &zrows,
                                ns.dead, prune ? sc->rmax_u.as<float>() : nullptr,
                                prune ? sc->rmin_u.as<float>() : nullptr, b,
                                prune ? sc->ext.as<unsigned int>() : nullptr);
        };
        {
            PhaseScope ph(m, AKASHIC_PHASE_SCORE, st);
            // with the row bounds (never with the dense fused filter) the
            // score GEMM's epilogue reduces u's row extremes into sc->ext,
            // zeroed here
            CUDA_TRY(launch_prep_queries(qb, b, bp, m->dim, m->tau, m->max_norm.as<float>(),
                                         sc->qp.as<uint16_t>(), sc->shift.as<float>(),
                                         m->status.as<int>(), st,
                                         prune ? sc->ext.as<unsigned int>() : nullptr));
            ph.launches += 1;
            if (reach_try)
                CUDA_TRY(launch_score_split(m->emb.as<uint16_t>(), n, m->dim,
                                            sc->qp.as<uint16_t>(), bp, sc->shift.as<float>(),
                                            m->tau, u_hi, u_lo, sc->zpart.as<float>(),
                                            m->status.as<int>(), st, &ph.launches, &zrows, ns.dead,
                                            sc->rmax_u.as<float>(), sc->rmin_u.as<float>(), b,
                                            sc->ext.as<unsigned int>()));
            else if (!dense_fused)
                CUDA_TRY(score_fp32(&ph.launches));
        }
        if (dense_fused) {
            {
                PhaseScope ps(m, AKASHIC_PHASE_SELECT, st);
                AK_TRY(ensure_spare(sc->samp, (size_t)sp.n_sample * bp * 4));
                AK_TRY(ensure_spare(sc->ext_s, (size_t)sp.n_sample * 4));
                AK_TRY(ensure_spare(sc->zsamp, (size_t)score_tiles(sp.n_sample) * bp * 4));
                CUDA_TRY(launch_ext_sample(m->ext_of.as<int32_t>(), sp.n_sample, sp.stride,
                                           sc->ext_s.as<int32_t>(), st));
                NsScope ns_samp{};
                if (q_ns) {
                    AK_TRY(ensure_spare(sc->ns_s, (size_t)sp.n_sample * 4));
                    CUDA_TRY(launch_ext_sample(m->ns_row.as<int32_t>(), sp.n_sample, sp.stride,
                                               sc->ns_s.as<int32_t>(), st));
                    ns_samp = NsScope{sc->ns_s.as<int32_t>(), sc->qns.as<int32_t>(), nullptr};
                }
                if (m->has_dead) {
                    AK_TRY(ensure_spare(sc->dead_s, (size_t)sp.n_sample * 4));
                    CUDA_TRY(launch_ext_sample(m->dead_row.as<int32_t>(), sp.n_sample, sp.stride,
                                               sc->dead_s.as<int32_t>(), st));
                    ns_samp.dead = sc->dead_s.as<int32_t>();
                }
                CUDA_TRY(launch_score_sample(m->emb.as<uint16_t>(), sp.n_sample, sp.stride, m->dim,
                                             sc->qp.as<uint16_t>(), bp, sc->shift.as<float>(),
                                             m->tau, sc->samp.as<float>(), sc->zsamp.as<float>(),
                                             m->status.as<int>(), st, &ps.launches));
                CUDA_TRY(launch_sample_bound(sp2, sc->samp.as<float>(), b, sc->ext_s.as<int32_t>(),
                                             ws, st, &ps.launches, 4u, ns_samp));
                ps.launches += 1;
            }
            PhaseScope ph(m, AKASHIC_PHASE_SCORE, st);
            CUDA_TRY(launch_score_filter(m->emb.as<uint16_t>(), n, m->dim, sc->qp.as<uint16_t>(),
                                         bp, b, sc->shift.as<float>(), m->tau,
                                         sc->zpart.as<float>(), m->ext_of.as<int32_t>(),
                                         ws + sp.off_bound, (unsigned int *)(ws + sp.off_cnt),
                                         ws + sp.off_buf, sp.cap, ns, m->status.as<int>(), st,
                                         &ph.launches, &zrows));
            rc.kind = 2;
            rc.emb = m->emb.as<uint16_t>();
            rc.qp = sc->qp.as<uint16_t>();
            rc.dim = m->dim;
            rc.tau = m->tau;
            rc.shift = sc->shift.as<float>();
            rc.dst = sc->u.as<float>();
        }
        const float *fin = sc->u.as<float>();
        if (eff_hops >= 1) {
            HopPlan hp;
            hp.split = m->split;
            hp.in_ptr = m->in_ptr.as<int64_t>();
            hp.in_src = m->in_src.as<int32_t>();
            hp.in_w = m->in_w.as<float>();
            hp.n = n;
            hp.n_split_rows = m->n_split;
            hp.split_row = m->split_row.as<int32_t>();
            hp.split_slot0 = m->split_slot0.as<int64_t>();
            hp.n_segs = m->n_segs;
            hp.seg_e0 = m->seg_e0.as<int64_t>();
            hp.seg_e1 = m->seg_e1.as<int64_t>();
            hp.seg_slot = m->seg_slot.as<int32_t>();
            hp.split_order = m->split_order.as<int32_t>();
            hp.slot_split = m->slot_split.as<int32_t>();
            float *bufs[2] = {sc->sa.as<float>(), sc->sb.as<float>()};
            rc.u = sc->u.as<float>();
            rc.in_ptr = hp.in_ptr;
            rc.in_src = hp.in_src;
            rc.in_w = hp.in_w;
            rc.alpha = alpha;
            // scalar row bounds of the last hop's output, from u's row extremes
            // (the two-hop reach path evaluates them only where it needs them
            // and writes the arrays only when the hops run after all)
            const float *row_ub = nullptr, *row_lb = nullptr;
            auto row_bounds = [&]() -> akashic_status_t {
                PhaseScope ph(m, AKASHIC_PHASE_BOUND, st);
                CUDA_TRY(launch_final_bounds(sc->rmax_u.as<float>(), sc->rmin_u.as<float>(),
                                             m->mass_up.as<float>(), m->mass_dn.as<float>(), n,
                                             eff_hops, alpha, sc->ext.as<unsigned int>(),
                                             sc->ub.as<float>(), sc->lb.as<float>(), st,
                                             &ph.launches, true));
                row_ub = sc->ub.as<float>();
                row_lb = sc->lb.as<float>();
                return AKASHIC_OK;
            };
            if (prune) {
                {
                    std::lock_guard<std::mutex> lk(m->table_mu);
                    AK_TRY(ensure_mass(m, hp, eff_hops, st));
                }
                if (!reach_try) AK_TRY(row_bounds());
            }
            // Two hops without running them: when every row whose upper bound
            // reaches the floor (here the k-th largest lower bound) is a
            // candidate with reach coefficients, their final scores come from
            // one pass over u and they alone are the selection's candidates.
            bool reach_done = false;
            if (reach_try) {
                {
                    PhaseScope ph(m, AKASHIC_PHASE_BOUND, st);
                    {
                        std::lock_guard<std::mutex> lk(m->table_mu);
                        AK_TRY(ensure_reach(m, hp, eff_hops, st));
                    }
                    AK_TRY(sc->reach_keep.ensure((REACH_T + 2) * 4));
                    AK_TRY(sc->reach_plan.ensure(REACH_PLAN_INTS * 4));
                    if (!sc->plan_host) CUDA_TRY(cudaMallocHost((void **)&sc->plan_host, 16));
                    if (!sc->plan_ev)
                        CUDA_TRY(cudaEventCreateWithFlags(&sc->plan_ev, cudaEventDisableTiming));
                    ReachFlags rf{};
                    rf.u0 = sc->rmax_u.as<float>();
                    rf.l0 = sc->rmin_u.as<float>();
                    rf.mup = m->mass_up.as<float>();
                    rf.mdn = m->mass_dn.as<float>();
                    rf.ext = sc->ext.as<unsigned int>();
                    rf.n = n;
                    rf.H = eff_hops;
                    rf.alpha = alpha;
                    rf.split_row = hp.split_row;
                    rf.split_order = hp.split_order;
                    rf.n_lb = m->n_split < 1024 ? m->n_split : 1024;
                    rf.k = k;
                    rf.map = m->reach_map.as<int32_t>();
                    rf.t_cnt = m->reach_t.as<int>();
                    rf.floor_out = sc->pfloor.as<float>();
                    rf.ws = sc->reach_keep.as<int32_t>();
                    rf.plan = sc->reach_plan.as<int32_t>();
                    CUDA_TRY(launch_reach_flags(rf, st, &ph.launches));
                    CUDA_TRY(cudaMemcpyAsync(sc->plan_host, sc->reach_plan.p, 8,
                                             cudaMemcpyDeviceToHost, st));
                    CUDA_TRY(cudaEventRecord(sc->plan_ev, st));
                }
                {
                    // The candidates' pass is queued before the host learns the
                    // plan (its kernels return at once when the plan says the
                    // hops run), so the GPU goes on while the host waits.
                    PhaseScope ph(m, AKASHIC_PHASE_LAST_HOP, st);
                    AK_TRY(sc->reach_part.ensure((size_t)reach_parts() * REACH_T * bp * 4));
                    // every candidate's packed coefficients, kept while the
                    // graph, alpha and the hop count stay the same
                    if (sc->coef_build != m->reach_build || sc->coef_alpha != alpha ||
                        sc->coef_H != eff_hops || sc->coef_n != n) {
                        const size_t cb = (size_t)REACH_T * reach_pad_rows(n) * 2;
                        AK_TRY(ensure_spare(sc->coef_hi, cb));
                        AK_TRY(ensure_spare(sc->coef_lo, cb));
                        CUDA_TRY(launch_reach_pack(m->reach_c.as<float>(), n, eff_hops, alpha,
                                                   sc->coef_hi.as<uint16_t>(),
                                                   sc->coef_lo.as<uint16_t>(), st));
                        ph.launches += 1;
                        sc->coef_build = m->reach_build;
                        sc->coef_alpha = alpha;
                        sc->coef_H = eff_hops;
                        sc->coef_n = n;
                    }
                    CUDA_TRY(launch_reach_scores(u_hi, u_lo, bp, b, n,
                                                 sc->coef_hi.as<uint16_t>(),
                                                 sc->coef_lo.as<uint16_t>(),
                                                 sc->reach_plan.as<int32_t>(),
                                                 m->reach_rows.as<int32_t>(),
                                                 m->ext_of.as<int32_t>(),
                                                 sc->reach_part.as<float>(),
                                                 (unsigned int *)(ws + sp.off_cnt), ws + sp.off_buf,
                                                 sp.cap, m->status.as<int>(), st, &ph.launches));
                }
                CUDA_TRY(cudaEventSynchronize(sc->plan_ev));
                if (sc->plan_host[0] == 1) {
                    rc = ColumnRecompute{};   // the buffers hold every candidate
                    reach_done = true;
                } else {
                    // the hops run: they read u in fp32 (the same scores again)
                    // and need every row's bounds
                    {
                        PhaseScope ph(m, AKASHIC_PHASE_SCORE, st);
                        CUDA_TRY(score_fp32(&ph.launches));
                    }
                    AK_TRY(row_bounds());
                }
            }
            for (int h = 0; h < eff_hops && !reach_done; ++h) {
                float *out = bufs[h & 1];
                const bool last = m->fuse_filter && h == eff_hops - 1;
                if (last) {
                    // Top-k filter fused into the last hop.  With w >= 0 and
                    // alpha >= 0 every hop only adds to a score, and in fp32
                    // too (same summation order, monotone rounding), so the
                    // k-th largest key of s^(H-1) over the row sample is a
                    // safe bound for s^(H).
                    {
                        PhaseScope ps(m, AKASHIC_PHASE_SELECT, st);
                        CUDA_TRY(launch_sample_bound(sp, fin, b, m->ext_of.as<int32_t>(), ws, st,
                                                     &ps.launches, 0u, ns));
                    }
                    if (prune) {
                        PhaseScope ps(m, AKASHIC_PHASE_BOUND, st);
                        // floor: the filter bounds', raised without a namespace
                        // scope to the k-th largest lower bound of the heaviest
                        // split rows (where the top scores lie)
                        const int64_t n_lb = m->n_split < 1024 ? m->n_split : 1024;
                        CUDA_TRY(launch_prune_floor(ws + sp.off_bound, b, row_lb,
                                                    q_ns ? nullptr : hp.split_row,
                                                    hp.split_order, n_lb, k,
                                                    sc->pfloor.as<float>(), st));
                        // with a scope, each namespace of the batch gets its own
                        // floor (its rows can only be selected by its queries)
                        NsFloors nf{};
                        if (q_ns) {
                            AK_TRY(sc->nsf.ensure(4096));
                            int32_t *tags = sc->nsf.as<int32_t>();
                            float *tag_floor = (float *)(tags + PF_TAGS);
                            int *n_tags = (int *)(tag_floor + PF_TAGS);
                            CUDA_TRY(launch_ns_floors(ws + sp.off_bound, sc->qns.as<int32_t>(), b,
                                                      row_lb, m->ns_row.as<int32_t>(),
                                                      hp.split_row, hp.split_order, m->n_split, k,
                                                      tags, n_tags, tag_floor, st));
                            nf = NsFloors{m->ns_row.as<int32_t>(), tags, n_tags, tag_floor};
                            ps.launches += m->n_split > 0 ? 2 : 1;
                        }
                        KeptScratch ks{sc->kflag.as<int64_t>(), sc->kpos.as<int64_t>(),
                                       sc->ktmp.p, sc->ktmp.cap};
                        CUDA_TRY(launch_split_flags(hp, row_ub, sc->pfloor.as<float>(),
                                                    q_ns ? &nf : nullptr,
                                                    sc->skip_split.as<int32_t>(),
                                                    sc->skip_slot.as<int32_t>(),
                                                    sc->kept_rows.as<int32_t>(),
                                                    sc->kept_count.as<int64_t>(),
                                                    sc->kept_segs.as<int32_t>(), ks, st,
                                                    &ps.launches));
                        ps.launches += 1;
                    }
                }
                const HopFilter flt{m->ext_of.as<int32_t>(), ws + sp.off_bound,
                                    (unsigned int *)(ws + sp.off_cnt), ws + sp.off_buf, sp.cap,
                                    ns};
                const HopBound hb{row_ub, sc->pfloor.as<float>(), sc->skip_split.as<int32_t>(),
                                  sc->skip_slot.as<int32_t>(), sc->kept_rows.as<int32_t>(),
                                  sc->kept_count.as<int64_t>(), sc->kept_segs.as<int32_t>()};
                PhaseScope ph(m, last ? AKASHIC_PHASE_LAST_HOP : AKASHIC_PHASE_PROPAGATE, st);
                CUDA_TRY(launch_hop(hp, sc->u.as<float>(), fin, out, bp, alpha,
                                    sc->partial.as<float>(), sc->counters.as<int>(),
                                    last ? &flt : nullptr, st, &ph.launches,
                                    (last && prune) ? &hb : nullptr));
                if (last) {
                    rc.kind = 1;
                    rc.prev = fin;
                    rc.dst = out;
                }
                fin = out;
            }
        }
        {
            PhaseScope ph(m, AKASHIC_PHASE_SELECT, st);
            int32_t *pids = page_ids ? page_ids + (int64_t)off * k : nullptr;
            int32_t *npg = n_pages ? n_pages + off : nullptr;
            if ((eff_hops >= 1 && m->fuse_filter) || dense_fused)
                CUDA_TRY(launch_topk_merge(sp, fin, b, sc->cand.as<unsigned long long>(),
                                           sc->zpart.as<float>(), zrows, m->ext_of.as<int32_t>(),
                                           m->row_of.as<int32_t>(), m->page_of.as<int32_t>(),
                                           ids + (int64_t)off * k, scores + (int64_t)off * k,
                                           pids, npg, m->status.as<int>(), &rc, ns,
                                           sort_by_time, st, &ph.launches));
            else
                CUDA_TRY(launch_select(sp, fin, b, sc->cand.as<unsigned long long>(),
                                       sc->zpart.as<float>(), zrows, m->ext_of.as<int32_t>(),
                                       m->row_of.as<int32_t>(), m->page_of.as<int32_t>(),
                                       ids + (int64_t)off * k, scores + (int64_t)off * k, pids,
                                       npg, m->status.as<int>(), ns, sort_by_time, st,
                                       &ph.launches));
        }
    }
    return AKASHIC_OK;
}

extern "C" {

akashic_status_t akashic_mem_export_csr(akashic_mem_t *m, int64_t *n_rows, int64_t *nnz,
                                        int64_t *row_ptr, int32_t *col, float *aff, float *w,
                                        void *stream) {
    g_last_error.clear();
    if (!m) return fail(AKASHIC_EINVAL, "export: NULL store");
    if (n_rows) *n_rows = m->n;
    if (nnz) *nnz = m->nnz;
    if (!row_ptr && !col && !aff && !w) return AKASHIC_OK;
    DeviceGuard g(m->device);
    cudaStream_t st = (cudaStream_t)stream;
    if (row_ptr)
        CUDA_TRY(cudaMemcpyAsync(row_ptr, m->row_ptr.p, (size_t)(m->n + 1) * 8,
                                 cudaMemcpyDeviceToDevice, st));
    if (m->nnz > 0) {
        if (col) CUDA_TRY(cudaMemcpyAsync(col, m->col.p, (size_t)m->nnz * 4, cudaMemcpyDeviceToDevice, st));
        if (aff) CUDA_TRY(cudaMemcpyAsync(aff, m->aff.p, (size_t)m->nnz * 4, cudaMemcpyDeviceToDevice, st));
        if (w) CUDA_TRY(cudaMemcpyAsync(w, m->w.p, (size_t)m->nnz * 4, cudaMemcpyDeviceToDevice, st));
    }
    CUDA_TRY(cudaStreamSynchronize(st));
    return AKASHIC_OK;
}

akashic_status_t akashic_mem_set_profiling(akashic_mem_t *m, int32_t on) {
    if (!m) return fail(AKASHIC_EINVAL, "set_profiling: NULL store");
    m->prof = on != 0;
    return AKASHIC_OK;
}

akashic_status_t akashic_mem_phase_times(akashic_mem_t *m, float *ms, int32_t *launches) {
    if (!m) return fail(AKASHIC_EINVAL, "phase_times: NULL store");
    DeviceGuard g(m->device);
    std::vector<ProfRec> recs;
    {
        std::lock_guard<std::mutex> lk(m->mu);
        recs.swap(m->recs);
    }
    for (int p = 0; p < AKASHIC_PHASE_COUNT; ++p) {
        if (ms) ms[p] = 0.f;
        if (launches) launches[p] = 0;
    }
    akashic_status_t rc = AKASHIC_OK;
    for (auto &r : recs) {
        float t = 0.f;
        cudaError_t e = cudaEventSynchronize(r.b);
        if (e == cudaSuccess) e = cudaEventElapsedTime(&t, r.a, r.b);
        if (e != cudaSuccess) {
            cudaGetLastError();
            rc = fail(AKASHIC_ECUDA, "phase_times: %s", cudaGetErrorString(e));
        }
        if (r.phase >= 0 && r.phase < AKASHIC_PHASE_COUNT) {
            if (ms) ms[r.phase] += t;
            if (launches) launches[r.phase] += r.launches;
        }
    }
    std::lock_guard<std::mutex> lk(m->mu);
    for (auto &r : recs) {
        m->ev_pool.push_back(r.a);
        m->ev_pool.push_back(r.b);
    }
    return rc;
}

}  // extern "C"
