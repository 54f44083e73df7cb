// Memory Manager on the device (arXiv 2607.05708, §4.2 and Algorithm 2):
// the page directory, co-retrieval statistics, association-driven
// relocation of retrieved chunks into fresh pages (out of place, old slots
// tombstoned) and compaction of pages whose invalid ratio reaches a
// threshold.  The paper's model calls have dense stand-ins:
//   affinity(a, b) = co(a, b) / (sel(a) + sel(b) - co(a, b)), the Jaccard
//     index of the request sets that retrieved a and b, "high association"
//     when co >= tau * (sel(a) + sel(b) - co) (fp64, tau rounded to fp32);
//   LLMCoLocate(S) = the chunks of S with a partner in S at or above tau;
//   LLMGroup(P) = connected components of those pairs within a namespace.
// A batch of requests adds its statistics first; its relocations then run
// in request order (one CTA walks the requests; lanes work on a request's
// chunk set).
#include "ak_common.cuh"

namespace ak {

constexpr unsigned long long MM_EMPTY = ~0ull;
constexpr int MM_MAX_S = 64;   // chunks per request set

// MurmurHash3's 64-bit finaliser (Appleby), spreading pair keys over the table.
__device__ __forceinline__ unsigned long long mm_mix(unsigned long long k) {
    k ^= k >> 33;
    k *= 0xff51afd7ed558ccdull;
    k ^= k >> 33;
    k *= 0xc4ceb9fe1a85ec53ull;
    k ^= k >> 33;
    return k;
}

__device__ __forceinline__ unsigned long long mm_pair(int32_t a, int32_t b) {
    const uint32_t lo = (uint32_t)(a < b ? a : b), hi = (uint32_t)(a < b ? b : a);
    return ((unsigned long long)lo << 32) | hi;
}

// co(a, b) += 1 (linear probing; a full table sets ECAPACITY)
__device__ void mm_co_add(const MmTables &t, unsigned long long key, int *status) {
    unsigned long long h = mm_mix(key) & (t.co_cap - 1);
    for (int64_t probe = 0; probe < t.co_cap; ++probe) {
        const unsigned long long prev = atomicCAS(&t.co_key[h], MM_EMPTY, key);
        if (prev == MM_EMPTY || prev == key) {
            atomicAdd(&t.co_val[h], 1u);
            return;
        }
        h = (h + 1) & (t.co_cap - 1);
    }
    set_status(status, AKASHIC_ECAPACITY);
}

__device__ uint32_t mm_co_get(const MmTables &t, unsigned long long key) {
    unsigned long long h = mm_mix(key) & (t.co_cap - 1);
    for (int64_t probe = 0; probe < t.co_cap; ++probe) {
        const unsigned long long k = t.co_key[h];
        if (k == key) return t.co_val[h];
        if (k == MM_EMPTY) return 0u;
        h = (h + 1) & (t.co_cap - 1);
    }
    return 0u;
}

__device__ __forceinline__ bool mm_assoc(uint32_t co, int32_t sa, int32_t sb, float tau) {
    const double uni = (double)sa + (double)sb - (double)co;
    return co > 0u && (double)co >= (double)tau * uni;
}

// The distinct valid chunks of request r (order of first appearance): IDs
// in [0, n), not deleted, first occurrence only.  Warp-cooperative; returns
// the count (same in every lane); set[] in shared memory.
__device__ int mm_request_set(const int64_t *__restrict__ S, int r, int s_len, int64_t n,
                              const int32_t *__restrict__ row_of,
                              const int32_t *__restrict__ dead_row, int32_t *set) {
    const int lane = threadIdx.x & 31;
    int32_t mine[2];
    bool ok[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int i = lane + 32 * h;
        int64_t c = i < s_len ? S[(int64_t)r * s_len + i] : -1;
        ok[h] = c >= 0 && c < n && !(dead_row && dead_row[row_of[c]]);
        mine[h] = ok[h] ? (int32_t)c : -1;
    }
    // drop repeats of an earlier position
    for (int j = 0; j < 32; ++j) {
        const int32_t o0 = __shfl_sync(0xffffffffu, mine[0], j);
        const int32_t o1 = __shfl_sync(0xffffffffu, mine[1], j);
        if (mine[0] >= 0 && j < lane && o0 == mine[0]) ok[0] = false;
        if (mine[1] >= 0 && (o0 == mine[1] || (j < lane && o1 == mine[1]))) ok[1] = false;
    }
    // compact the survivors in position order
    int count = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const unsigned m = __ballot_sync(0xffffffffu, ok[h]);
        if (ok[h]) set[count + __popc(m & ((1u << lane) - 1u))] = mine[h];
        count += __popc(m);
    }
    __syncwarp();
    return count;
}

// Statistics of a batch: one warp per request.
__global__ void k_mm_count(const int64_t *__restrict__ S, int n_req, int s_len, int64_t n,
                           const int32_t *__restrict__ row_of,
                           const int32_t *__restrict__ dead_row, MmTables t, int *status) {
    __shared__ int32_t sets[8][MM_MAX_S];
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int r = blockIdx.x * 8 + w; r < n_req; r += gridDim.x * 8) {
        const int cnt = mm_request_set(S, r, s_len, n, row_of, dead_row, sets[w]);
        for (int i = lane; i < cnt; i += 32) atomicAdd(&t.sel[sets[w][i]], 1);
        for (int p = lane; p < cnt * cnt; p += 32) {
            const int i = p / cnt, j = p % cnt;
            if (i < j) mm_co_add(t, mm_pair(sets[w][i], sets[w][j]), status);
        }
        __syncwarp();
    }
}

// LLMCoLocate stand-in for every request of the batch (the statistics of
// the whole batch are in place): G = the chunks of the set associated with
// some other chunk of it, in chunk ID order.  One warp per request.
__global__ void k_mm_colocate(const int64_t *__restrict__ S, int n_req, int s_len, int64_t n,
                              const int32_t *__restrict__ row_of,
                              const int32_t *__restrict__ dead_row, MmTables t, float tau,
                              int32_t *__restrict__ g_out, int32_t *__restrict__ g_n) {
    __shared__ int32_t sets[8][MM_MAX_S];
    __shared__ int flags[8][MM_MAX_S];
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int r = blockIdx.x * 8 + w; r < n_req; r += gridDim.x * 8) {
        const int cnt = mm_request_set(S, r, s_len, n, row_of, dead_row, sets[w]);
        for (int i = lane; i < MM_MAX_S; i += 32) flags[w][i] = 0;
        __syncwarp();
        for (int p = lane; p < cnt * cnt; p += 32) {
            const int i = p / cnt, j = p % cnt;
            if (i >= j) continue;
            const int32_t a = sets[w][i], b = sets[w][j];
            if (mm_assoc(mm_co_get(t, mm_pair(a, b)), t.sel[a], t.sel[b], tau)) {
                flags[w][i] = 1;
                flags[w][j] = 1;
            }
        }
        __syncwarp();
        int ng = 0;
        for (int i = 0; i < cnt; ++i) ng += flags[w][i];
        // G in chunk ID order (SortByTime): rank by counting
        for (int i = lane; i < cnt; i += 32) {
            if (!flags[w][i]) continue;
            const int32_t a = sets[w][i];
            int rk = 0;
            for (int j = 0; j < cnt; ++j) rk += flags[w][j] && sets[w][j] < a;
            g_out[(int64_t)r * MM_MAX_S + rk] = a;
        }
        if (lane == 0) g_n[r] = ng;
        __syncwarp();
    }
}

// Relocation in request order (one warp): a G of two or more chunks not all
// on one page is written into fresh pages, old slots become invalid.
__global__ void k_mm_relocate(const int32_t *__restrict__ g_in, const int32_t *__restrict__ g_n,
                              int n_req, const int32_t *__restrict__ row_of,
                              int32_t *__restrict__ page_row, MmTables t, int per_page) {
    const int lane = threadIdx.x & 31;
    int64_t next = *t.next_page;
    int64_t writes = 0;
    for (int r = 0; r < n_req; ++r) {
        const int ng = g_n[r];
        if (ng < 2) continue;
        const int32_t *g = g_in + (int64_t)r * MM_MAX_S;
        const int32_t p0 = page_row[row_of[g[0]]];
        bool same = true;
        for (int i = lane; i < ng; i += 32) same &= page_row[row_of[g[i]]] == p0;
        if (__all_sync(0xffffffffu, same)) continue;
        __syncwarp();
        for (int i = lane; i < ng; i += 32) {
            const int64_t row = row_of[g[i]];
            atomicSub(&t.page_live[page_row[row]], 1);
            const int32_t p = (int32_t)(next + i / per_page);
            page_row[row] = p;
            atomicAdd(&t.page_total[p], 1);
            atomicAdd(&t.page_live[p], 1);
        }
        __syncwarp();
        next += (ng + per_page - 1) / per_page;
        writes += ng;
    }
    if (lane == 0) {
        *t.next_page = next;
        *t.writes += writes;
    }
}

// ------------------------------------------------------------------ compaction
__global__ void k_mm_candidates(MmTables t, int64_t n_pages, float theta, int32_t *__restrict__ cand) {
    // warp-uniform trip count, so the whole warp takes part in every ballot
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t base = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); base < n_pages;
         base += stride) {
        const int64_t p = base + (threadIdx.x & 31);
        bool c = false;
        if (p < n_pages) {
            const int32_t tot = t.page_total[p], live = t.page_live[p];
            c = tot > 0 && (double)(tot - live) >= (double)theta * (double)tot;
            cand[p] = c;
        }
        const unsigned ballot = __ballot_sync(0xffffffffu, c);
        if ((threadIdx.x & 31) == 0 && ballot) atomicAdd(t.released, (unsigned long long)__popc(ballot));
    }
}

// moving[c] = 1 for live chunks on candidate pages; parent[c] = c
__global__ void k_mm_moving(int64_t n, const int32_t *__restrict__ row_of,
                            const int32_t *__restrict__ dead_row,
                            const int32_t *__restrict__ page_row, const int32_t *__restrict__ cand,
                            int64_t *__restrict__ moving, int32_t *__restrict__ parent) {
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < n;
         c += (int64_t)gridDim.x * blockDim.x) {
        const int64_t row = row_of[c];
        const bool mv = !(dead_row && dead_row[row]) && cand[page_row[row]];
        moving[c] = mv ? 1 : 0;
        parent[c] = (int32_t)c;
    }
}

__device__ int32_t mm_find(volatile int32_t *parent, int32_t x) {
    for (int it = 0; it < (1 << 24); ++it) {
        const int32_t p = parent[x];
        if (p == x) return x;
        x = p;
    }
    return x;
}

// union of every associated pair of moving chunks in one namespace; roots
// hook under the smaller root, so a group's root is its earliest chunk
__global__ void k_mm_union(MmTables t, const int64_t *__restrict__ moving,
                           const int32_t *__restrict__ ns_by_id, float tau,
                           int32_t *__restrict__ parent, int *status) {
    for (int64_t h = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; h < t.co_cap;
         h += (int64_t)gridDim.x * blockDim.x) {
        const unsigned long long key = t.co_key[h];
        if (key == MM_EMPTY) continue;
        const int32_t a = (int32_t)(key >> 32), b = (int32_t)(key & 0xffffffffu);
        if (!moving[a] || !moving[b] || ns_by_id[a] != ns_by_id[b]) continue;
        if (!mm_assoc(t.co_val[h], t.sel[a], t.sel[b], tau)) continue;
        volatile int32_t *vp = parent;
        int it = 0;
        for (; it < (1 << 20); ++it) {
            const int32_t ra = mm_find(vp, a), rb = mm_find(vp, b);
            if (ra == rb) break;
            const int32_t hi = ra > rb ? ra : rb, lo = ra > rb ? rb : ra;
            if (atomicCAS(&parent[hi], hi, lo) == hi) break;
        }
        if (it == (1 << 20)) set_status(status, AKASHIC_ETIMEOUT);
    }
}

// keys for the ordered repack: (namespace, group root, chunk ID); the
// moving chunks arrive in ID order (compacted by scan)
__global__ void k_mm_keys(const int64_t *__restrict__ moving, const int64_t *__restrict__ pos,
                          int64_t n, const int32_t *__restrict__ parent,
                          const int32_t *__restrict__ ns_by_id, uint32_t *__restrict__ ids,
                          uint32_t *__restrict__ root_key, uint32_t *__restrict__ ns_key) {
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < n;
         c += (int64_t)gridDim.x * blockDim.x) {
        if (!moving[c]) continue;
        const int64_t i = pos[c];
        ids[i] = (uint32_t)c;
        root_key[i] = (uint32_t)mm_find((volatile int32_t *)parent, (int32_t)c);
        ns_key[i] = (uint32_t)ns_by_id[c] ^ 0x80000000u;   // signed order
    }
}

__global__ void k_mm_ns_keys(const uint32_t *__restrict__ ids, int64_t count,
                             const int32_t *__restrict__ ns_by_id, uint32_t *__restrict__ out) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count;
         i += (int64_t)gridDim.x * blockDim.x)
        out[i] = (uint32_t)ns_by_id[ids[i]] ^ 0x80000000u;
}

cudaError_t launch_mm_ns_keys(const uint32_t *ids, int64_t count, const int32_t *ns_by_id,
                              uint32_t *out, cudaStream_t st) {
    if (count <= 0) return cudaSuccess;
    k_mm_ns_keys<<<device_sm_count() * 2, 256, 0, st>>>(ids, count, ns_by_id, out);
    return cudaGetLastError();
}

__global__ void k_mm_release(MmTables t, int64_t n_pages, const int32_t *__restrict__ cand) {
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < n_pages;
         p += (int64_t)gridDim.x * blockDim.x)
        if (cand[p]) {
            t.page_total[p] = 0;
            t.page_live[p] = 0;
        }
}

// first index of the sorted keys[0, count) holding a key >= v
__device__ __forceinline__ int64_t lower_bound_u32(const uint32_t *__restrict__ keys, int64_t count,
                                                   uint32_t v) {
    int64_t lo = 0, hi = count;
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if (keys[mid] < v) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

// Every namespace (partition) starts on a fresh page: at the first
// position of each run of equal namespace keys, the pages that run fills
// (ceil(run / P)); zero elsewhere.  An exclusive scan of these gives each
// partition's first page relative to the first fresh page.
__global__ void k_mm_part_pages(const uint32_t *__restrict__ ns_sorted, int64_t count,
                                int per_page, int64_t *__restrict__ part_pages) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count;
         i += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t k = ns_sorted[i];
        int64_t v = 0;
        if (i == 0 || ns_sorted[i - 1] != k) {
            const int64_t end = k == 0xffffffffu ? count : lower_bound_u32(ns_sorted, count, k + 1);
            v = (end - i + per_page - 1) / per_page;
        }
        part_pages[i] = v;
    }
}

cudaError_t launch_mm_part_pages(const uint32_t *ns_sorted, int64_t count, int per_page,
                                 int64_t *part_pages, cudaStream_t st) {
    if (count <= 0) return cudaSuccess;
    k_mm_part_pages<<<device_sm_count() * 2, 256, 0, st>>>(ns_sorted, count, per_page, part_pages);
    return cudaGetLastError();
}

// chunk i of the ordered list: page = first page + its partition's base
// page + (offset inside the partition) / P
__global__ void k_mm_repack(const uint32_t *__restrict__ order_ids,
                            const uint32_t *__restrict__ ns_sorted,
                            const int64_t *__restrict__ part_base, int64_t count,
                            const int32_t *__restrict__ row_of, int32_t *__restrict__ page_row,
                            MmTables t, int64_t first_page, int per_page) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t s = lower_bound_u32(ns_sorted, count, ns_sorted[i]);
        const int32_t p = (int32_t)(first_page + part_base[s] + (i - s) / per_page);
        page_row[row_of[order_ids[i]]] = p;
        atomicAdd(&t.page_total[p], 1);
        atomicAdd(&t.page_live[p], 1);
    }
}

// ------------------------------------------------------------------ bookkeeping
// new rows [first, first+n): their pages gain a live slot each
__global__ void k_mm_count_pages(const int32_t *__restrict__ page_row, int64_t first, int64_t n,
                                 MmTables t) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int32_t p = page_row[first + i];
        atomicAdd(&t.page_total[p], 1);
        atomicAdd(&t.page_live[p], 1);
    }
}

__global__ void k_mm_stats(MmTables t, int64_t n_pages, unsigned long long *__restrict__ out) {
    unsigned long long in_use = 0, tot = 0, live = 0;
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < n_pages;
         p += (int64_t)gridDim.x * blockDim.x) {
        const int32_t a = t.page_total[p];
        in_use += a > 0;
        tot += (unsigned long long)(a > 0 ? a : 0);
        live += (unsigned long long)(a > 0 ? t.page_live[p] : 0);
    }
    for (int o = 16; o > 0; o >>= 1) {
        in_use += __shfl_xor_sync(0xffffffffu, in_use, o);
        tot += __shfl_xor_sync(0xffffffffu, tot, o);
        live += __shfl_xor_sync(0xffffffffu, live, o);
    }
    if ((threadIdx.x & 31) == 0) {
        atomicAdd(&out[0], in_use);
        atomicAdd(&out[1], tot);
        atomicAdd(&out[2], live);
    }
}

__global__ void k_mm_rehash(const unsigned long long *__restrict__ old_key,
                            const uint32_t *__restrict__ old_val, int64_t old_cap, MmTables t,
                            int *status) {
    for (int64_t h = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; h < old_cap;
         h += (int64_t)gridDim.x * blockDim.x) {
        const unsigned long long key = old_key[h];
        if (key == MM_EMPTY) continue;
        unsigned long long j = mm_mix(key) & (t.co_cap - 1);
        int64_t probe = 0;
        for (; probe < t.co_cap; ++probe) {
            if (atomicCAS(&t.co_key[j], MM_EMPTY, key) == MM_EMPTY) {
                t.co_val[j] = old_val[h];
                break;
            }
            j = (j + 1) & (t.co_cap - 1);
        }
        if (probe == t.co_cap) set_status(status, AKASHIC_ECAPACITY);
    }
}

__global__ void k_by_id(const int32_t *__restrict__ by_row, const int32_t *__restrict__ row_of,
                        int64_t n, int32_t *__restrict__ out) {
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < n;
         c += (int64_t)gridDim.x * blockDim.x)
        out[c] = by_row[row_of[c]];
}

// ------------------------------------------------------------------ launchers
cudaError_t launch_mm_count(const int64_t *S, int n_req, int s_len, int64_t n,
                            const int32_t *row_of, const int32_t *dead_row, const MmTables &t,
                            int *status, cudaStream_t st) {
    if (n_req <= 0) return cudaSuccess;
    const int grid = (int)ceil_div<int64_t>(n_req, 8);
    k_mm_count<<<grid < device_sm_count() * 8 ? grid : device_sm_count() * 8, 256, 0, st>>>(
        S, n_req, s_len, n, row_of, dead_row, t, status);
    return cudaGetLastError();
}

cudaError_t launch_mm_relocate(const int64_t *S, int n_req, int s_len, int64_t n,
                               const int32_t *row_of, const int32_t *dead_row, int32_t *page_row,
                               const MmTables &t, float tau, int per_page, int32_t *g_buf,
                               int32_t *g_n, cudaStream_t st) {
    if (n_req <= 0) return cudaSuccess;
    const int grid = (int)ceil_div<int64_t>(n_req, 8);
    k_mm_colocate<<<grid < device_sm_count() * 8 ? grid : device_sm_count() * 8, 256, 0, st>>>(
        S, n_req, s_len, n, row_of, dead_row, t, tau, g_buf, g_n);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_mm_relocate<<<1, 32, 0, st>>>(g_buf, g_n, n_req, row_of, page_row, t, per_page);
    return cudaGetLastError();
}

cudaError_t launch_mm_compact_prepare(const MmTables &t, int64_t n_pages, float theta, int64_t n,
                                      const int32_t *row_of, const int32_t *dead_row,
                                      const int32_t *page_row, int32_t *cand, int64_t *moving,
                                      int32_t *parent, cudaStream_t st) {
    const int sms = device_sm_count();
    if (n_pages > 0) k_mm_candidates<<<sms * 2, 256, 0, st>>>(t, n_pages, theta, cand);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || n <= 0) return e;
    k_mm_moving<<<sms * 4, 256, 0, st>>>(n, row_of, dead_row, page_row, cand, moving, parent);
    return cudaGetLastError();
}

cudaError_t launch_mm_union(const MmTables &t, const int64_t *moving, const int32_t *ns_by_id,
                            float tau, int32_t *parent, int *status, cudaStream_t st) {
    k_mm_union<<<device_sm_count() * 8, 256, 0, st>>>(t, moving, ns_by_id, tau, parent, status);
    return cudaGetLastError();
}

cudaError_t launch_mm_keys(const int64_t *moving, const int64_t *pos, int64_t n,
                           const int32_t *parent, const int32_t *ns_by_id, uint32_t *ids,
                           uint32_t *root_key, uint32_t *ns_key, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_mm_keys<<<device_sm_count() * 4, 256, 0, st>>>(moving, pos, n, parent, ns_by_id, ids,
                                                     root_key, ns_key);
    return cudaGetLastError();
}

cudaError_t launch_mm_release_repack(const MmTables &t, int64_t n_pages, const int32_t *cand,
                                     const uint32_t *order_ids, const uint32_t *ns_sorted,
                                     const int64_t *part_base, int64_t count,
                                     const int32_t *row_of, int32_t *page_row, int64_t first_page,
                                     int per_page, cudaStream_t st) {
    const int sms = device_sm_count();
    if (n_pages > 0) k_mm_release<<<sms * 2, 256, 0, st>>>(t, n_pages, cand);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || count <= 0) return e;
    k_mm_repack<<<sms * 2, 256, 0, st>>>(order_ids, ns_sorted, part_base, count, row_of, page_row,
                                         t, first_page, per_page);
    return cudaGetLastError();
}

cudaError_t launch_mm_count_pages(const int32_t *page_row, int64_t first, int64_t n,
                                  const MmTables &t, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_mm_count_pages<<<device_sm_count() * 2, 256, 0, st>>>(page_row, first, n, t);
    return cudaGetLastError();
}

cudaError_t launch_mm_stats(const MmTables &t, int64_t n_pages, unsigned long long *out,
                            cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(out, 0, 3 * sizeof(unsigned long long), st);
    if (e != cudaSuccess || n_pages <= 0) return e;
    k_mm_stats<<<device_sm_count() * 2, 256, 0, st>>>(t, n_pages, out);
    return cudaGetLastError();
}

cudaError_t launch_mm_rehash(const unsigned long long *old_key, const uint32_t *old_val,
                             int64_t old_cap, const MmTables &t, int *status, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(t.co_key, 0xff, (size_t)t.co_cap * 8, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(t.co_val, 0, (size_t)t.co_cap * 4, st);
    if (e != cudaSuccess || old_cap <= 0) return e;
    k_mm_rehash<<<device_sm_count() * 8, 256, 0, st>>>(old_key, old_val, old_cap, t, status);
    return cudaGetLastError();
}

cudaError_t launch_by_id(const int32_t *by_row, const int32_t *row_of, int64_t n, int32_t *out,
                         cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_by_id<<<device_sm_count() * 2, 256, 0, st>>>(by_row, row_of, n, out);
    return cudaGetLastError();
}

}  // namespace ak
