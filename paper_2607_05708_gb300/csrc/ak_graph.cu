// Relation graph on the device: prefix sums, a stable LSD radix sort, the
// in-edge transpose in store-row space, relation weights, the page-order
// layout of appended chunks, and the propagation hop (a2) that
// spreads scores along cross-chunk relations (arXiv 2607.05708, §4.1:
// related chunks are recovered together).
#include "ak_common.cuh"

namespace ak {

static int sm_count_cached() {
    static int cached[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) dev = 0;
    if (!cached[dev]) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        cached[dev] = v > 0 ? v : 1;
    }
    return cached[dev];
}
int device_sm_count() { return sm_count_cached(); }

// ================================================================== scan
constexpr int SCAN_THREADS = 256, SCAN_ITEMS = 8, SCAN_TILE = SCAN_THREADS * SCAN_ITEMS;

__device__ __forceinline__ int64_t warp_incl_scan(int64_t v) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int64_t t = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += t;
    }
    return v;
}

// Each CTA scans one tile of SCAN_TILE values (exclusive) and emits the
// tile total.
__global__ __launch_bounds__(SCAN_THREADS) void k_scan_tile(const int64_t *__restrict__ in,
                                                            int64_t *__restrict__ out, int64_t n,
                                                            int64_t *__restrict__ tile_sum) {
    __shared__ int64_t wsum[SCAN_THREADS / 32];
    const int64_t base = (int64_t)blockIdx.x * SCAN_TILE + (int64_t)threadIdx.x * SCAN_ITEMS;
    int64_t v[SCAN_ITEMS];
    int64_t run = 0;
#pragma unroll
    for (int i = 0; i < SCAN_ITEMS; ++i) {
        int64_t idx = base + i;
        v[i] = idx < n ? in[idx] : 0;
        run += v[i];
    }
    int64_t incl = warp_incl_scan(run);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        int64_t s = lane < SCAN_THREADS / 32 ? wsum[lane] : 0;
        s = warp_incl_scan(s);
        if (lane < SCAN_THREADS / 32) wsum[lane] = s;
    }
    __syncthreads();
    int64_t excl = incl - run + (warp > 0 ? wsum[warp - 1] : 0);
#pragma unroll
    for (int i = 0; i < SCAN_ITEMS; ++i) {
        int64_t idx = base + i;
        if (idx < n) out[idx] = excl;
        excl += v[i];
    }
    if (threadIdx.x == SCAN_THREADS - 1) tile_sum[blockIdx.x] = excl;
}

__global__ void k_scan_add(int64_t *__restrict__ out, int64_t n,
                           const int64_t *__restrict__ tile_off) {
    int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx < n) out[idx] += tile_off[idx / SCAN_TILE];
}

__global__ void k_scan_total(const int64_t *__restrict__ in, int64_t *__restrict__ out,
                             int64_t n) {
    // out[n] = out[n-1] + in[n-1]  (n >= 1), else 0
    out[n] = n > 0 ? out[n - 1] + in[n - 1] : 0;
}

// Flat form, for at most SCAN_FLAT_TILES tiles: the tile sums, then each CTA
// adds up the sums of the tiles before it and scans its own tile; the last
// CTA writes the total.  Two launches (one for a single tile).
constexpr int64_t SCAN_FLAT_TILES = 1024;

__device__ __forceinline__ int64_t block_sum_scan(int64_t v, int64_t *wsum) {
    // the CTA's sum of v, on every thread (wsum: SCAN_THREADS / 32 slots)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) wsum[warp] = v;
    __syncthreads();
    int64_t s = 0;
#pragma unroll
    for (int w = 0; w < SCAN_THREADS / 32; ++w) s += wsum[w];
    return s;
}

__global__ __launch_bounds__(SCAN_THREADS) void k_scan_reduce(const int64_t *__restrict__ in,
                                                              int64_t n,
                                                              int64_t *__restrict__ tile_sum) {
    __shared__ int64_t wsum[SCAN_THREADS / 32];
    const int64_t base = (int64_t)blockIdx.x * SCAN_TILE;
    int64_t s = 0;
#pragma unroll
    for (int i = 0; i < SCAN_ITEMS; ++i) {
        const int64_t idx = base + i * SCAN_THREADS + threadIdx.x;
        if (idx < n) s += in[idx];
    }
    s = block_sum_scan(s, wsum);
    if (threadIdx.x == 0) tile_sum[blockIdx.x] = s;
}

__global__ __launch_bounds__(SCAN_THREADS) void k_scan_down(const int64_t *__restrict__ in,
                                                            int64_t *__restrict__ out, int64_t n,
                                                            const int64_t *__restrict__ tile_sum) {
    __shared__ int64_t wsum[SCAN_THREADS / 32];
    int64_t pre = 0;
    for (int64_t t = threadIdx.x; t < (int64_t)blockIdx.x; t += SCAN_THREADS) pre += tile_sum[t];
    pre = block_sum_scan(pre, wsum);
    __syncthreads();   // wsum is reused below
    const int64_t base = (int64_t)blockIdx.x * SCAN_TILE + (int64_t)threadIdx.x * SCAN_ITEMS;
    int64_t v[SCAN_ITEMS];
    int64_t run = 0;
#pragma unroll
    for (int i = 0; i < SCAN_ITEMS; ++i) {
        const int64_t idx = base + i;
        v[i] = idx < n ? in[idx] : 0;
        run += v[i];
    }
    const int64_t incl = warp_incl_scan(run);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    int64_t excl = pre + incl - run;
    for (int w = 0; w < warp; ++w) excl += wsum[w];
#pragma unroll
    for (int i = 0; i < SCAN_ITEMS; ++i) {
        const int64_t idx = base + i;
        if (idx < n) out[idx] = excl;
        excl += v[i];
    }
    if (blockIdx.x == gridDim.x - 1 && threadIdx.x == SCAN_THREADS - 1) out[n] = excl;
}

size_t scan_tmp_bytes(int64_t n) {
    size_t tot = 0;
    int64_t m = n;
    do {
        int64_t tiles = ceil_div<int64_t>(m, SCAN_TILE);
        tot += (size_t)(2 * tiles + 2) * sizeof(int64_t);
        m = tiles;
    } while (m > 1);
    return tot + 64;
}

static cudaError_t scan_rec(const int64_t *in, int64_t *out, int64_t n, int64_t *tmp,
                            cudaStream_t st, int *launches) {
    if (n <= 0) return cudaSuccess;
    int64_t tiles = ceil_div<int64_t>(n, SCAN_TILE);
    int64_t *sums = tmp, *offs = tmp + tiles;
    k_scan_tile<<<(unsigned)tiles, SCAN_THREADS, 0, st>>>(in, out, n, sums);
    if (launches) *launches += 1;
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || tiles == 1) return e;
    e = scan_rec(sums, offs, tiles, tmp + 2 * tiles + 2, st, launches);
    if (e != cudaSuccess) return e;
    k_scan_add<<<(unsigned)ceil_div<int64_t>(n, 256), 256, 0, st>>>(out, n, offs);
    if (launches) *launches += 1;
    return cudaGetLastError();
}

cudaError_t scan_exclusive(const int64_t *in, int64_t *out, int64_t n, void *tmp,
                           size_t tmp_bytes, cudaStream_t st, int *launches) {
    if (tmp_bytes < scan_tmp_bytes(n)) return cudaErrorInvalidValue;
    const int64_t tiles = ceil_div<int64_t>(n, SCAN_TILE);
    if (n > 0 && tiles <= SCAN_FLAT_TILES) {
        int64_t *sums = (int64_t *)tmp;
        if (tiles > 1) k_scan_reduce<<<(unsigned)tiles, SCAN_THREADS, 0, st>>>(in, n, sums);
        k_scan_down<<<(unsigned)tiles, SCAN_THREADS, 0, st>>>(in, out, n, sums);
        if (launches) *launches += tiles > 1 ? 2 : 1;
        return cudaGetLastError();
    }
    cudaError_t e = scan_rec(in, out, n, (int64_t *)tmp, st, launches);
    if (e != cudaSuccess) return e;
    k_scan_total<<<1, 1, 0, st>>>(in, out, n);
    if (launches) *launches += 1;
    return cudaGetLastError();
}

// ================================================================== radix sort
// Stable LSD radix sort of (uint32 key, uint32 value) pairs, 8 bits a pass.
// Per pass: tile histograms (digit-major), one exclusive scan, then a stable
// scatter in which each warp ranks its keys round by round with
// __match_any_sync and the warps of a tile are combined in order.
constexpr int RS_THREADS = 256, RS_ITEMS = 16, RS_TILE = RS_THREADS * RS_ITEMS;
constexpr int RS_WARPS = RS_THREADS / 32, RS_PER_WARP = RS_TILE / RS_WARPS;

__global__ __launch_bounds__(RS_THREADS) void k_rs_hist(const uint32_t *__restrict__ keys,
                                                        int64_t n, int shift, uint32_t mask,
                                                        int64_t n_tiles,
                                                        int64_t *__restrict__ hist) {
    __shared__ int h[256];
    h[threadIdx.x] = 0;
    __syncthreads();
    const int64_t base = (int64_t)blockIdx.x * RS_TILE;
    for (int i = threadIdx.x; i < RS_TILE; i += RS_THREADS) {
        int64_t idx = base + i;
        if (idx < n) atomicAdd(&h[(keys[idx] >> shift) & mask], 1);
    }
    __syncthreads();
    hist[(int64_t)threadIdx.x * n_tiles + blockIdx.x] = h[threadIdx.x];
}

// Rank the warp's 32 * ITEMS keys of the tile stably by digit: loc[r] is
// the key's rank among the warp's keys of its digit, cnt[warp][d] the
// warp's count of digit d; then pre[w][d] = the counts of digit d in the
// warps before w (one thread a digit).  Keys at or past n get no digit.
template <int ITEMS>
__device__ __forceinline__ void rs_rank(const uint32_t *__restrict__ keys,
                                        const uint32_t *__restrict__ vals, int64_t n,
                                        int64_t base, int shift, uint32_t mask,
                                        uint32_t (&k)[ITEMS], uint32_t (&v)[ITEMS],
                                        int (&loc)[ITEMS], int (*cnt)[256], int (*pre)[256]) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int d = lane; d < 256; d += 32) cnt[warp][d] = 0;
    __syncwarp();
    const unsigned lt = (1u << lane) - 1u;
    // every load first, then the ranking (whose rounds depend on each other)
#pragma unroll
    for (int r = 0; r < ITEMS; ++r) {
        const int64_t idx = base + r * 32 + lane;
        k[r] = idx < n ? keys[idx] : 0u;
        v[r] = idx < n ? vals[idx] : 0u;
    }
#pragma unroll
    for (int r = 0; r < ITEMS; ++r) {
        int64_t idx = base + r * 32 + lane;
        bool ok = idx < n;
        uint32_t d = ok ? ((k[r] >> shift) & mask) : 0x100u;   // 0x100: no digit
        unsigned peers = __match_any_sync(0xffffffffu, d);
        int leader = __ffs(peers) - 1;
        int c = ok ? cnt[warp][d] : 0;
        loc[r] = c + __popc(peers & lt);
        __syncwarp();
        if (ok && lane == leader) cnt[warp][d] = c + __popc(peers);
        __syncwarp();
    }
    __syncthreads();
    {
        int d = threadIdx.x;   // RS_THREADS == 256 digits
        int run = 0;
#pragma unroll
        for (int w = 0; w < RS_WARPS; ++w) {
            pre[w][d] = run;
            run += cnt[w][d];
        }
    }
    __syncthreads();
}

__global__ __launch_bounds__(RS_THREADS) void k_rs_scatter(
    const uint32_t *__restrict__ keys, const uint32_t *__restrict__ vals, int64_t n, int shift,
    uint32_t mask, int64_t n_tiles, const int64_t *__restrict__ offs, uint32_t *__restrict__ okeys,
    uint32_t *__restrict__ ovals) {
    __shared__ int cnt[RS_WARPS][256];
    __shared__ int pre[RS_WARPS][256];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t base = (int64_t)blockIdx.x * RS_TILE + (int64_t)warp * RS_PER_WARP;
    uint32_t k[RS_ITEMS], v[RS_ITEMS];
    int loc[RS_ITEMS];
    rs_rank<RS_ITEMS>(keys, vals, n, base, shift, mask, k, v, loc, cnt, pre);
#pragma unroll
    for (int r = 0; r < RS_ITEMS; ++r) {
        int64_t idx = base + r * 32 + lane;
        if (idx < n) {
            uint32_t d = (k[r] >> shift) & mask;
            int64_t pos = offs[(int64_t)d * n_tiles + blockIdx.x] + pre[warp][d] + loc[r];
            okeys[pos] = k[r];
            ovals[pos] = v[r];
        }
    }
}

// Small sorts (at most RS_SMALL_TILES tiles of RS_SMALL_TILE keys: four a
// thread, so that a sort of ~100k pairs still spreads over ~100 CTAs) take
// one launch a pass after a first histogram launch.  Histograms are int32,
// digit-major [256][n_tiles].
// Each scatter CTA derives its own offsets from the pass's histograms (the
// totals of the smaller digits plus its digit's counts in the tiles before
// it) and counts the next pass's digit of every key it places into the next
// histograms, by destination tile.  Three histogram buffers rotate: pass p
// reads H[p % 3], counts into H[(p+1) % 3] (zero by then) and zeroes its
// column of H[(p+2) % 3], which pass p-1 read and pass p+1 counts into.
constexpr int RS_SMALL_ITEMS = 4, RS_SMALL_TILE = RS_THREADS * RS_SMALL_ITEMS;
constexpr int64_t RS_SMALL_TILES = 256;

__global__ __launch_bounds__(RS_THREADS) void k_rs_hist32(const uint32_t *__restrict__ keys,
                                                          int64_t n, int shift, uint32_t mask,
                                                          int n_tiles, int *__restrict__ hist,
                                                          int *__restrict__ zero1,
                                                          int *__restrict__ zero2) {
    __shared__ int h[256];
    h[threadIdx.x] = 0;
    __syncthreads();
    const int64_t base = (int64_t)blockIdx.x * RS_SMALL_TILE;
    for (int i = threadIdx.x; i < RS_SMALL_TILE; i += RS_THREADS) {
        int64_t idx = base + i;
        if (idx < n) atomicAdd(&h[(keys[idx] >> shift) & mask], 1);
    }
    __syncthreads();
    const int64_t at = (int64_t)threadIdx.x * n_tiles + blockIdx.x;
    hist[at] = h[threadIdx.x];
    zero1[at] = 0;
    zero2[at] = 0;
}

__global__ __launch_bounds__(RS_THREADS) void k_rs_scatter_small(
    const uint32_t *__restrict__ keys, const uint32_t *__restrict__ vals, int64_t n, int shift,
    uint32_t mask, int n_tiles, const int *__restrict__ hcur, int *__restrict__ hnext,
    int shift_next, uint32_t mask_next, int *__restrict__ hzero, uint32_t *__restrict__ okeys,
    uint32_t *__restrict__ ovals) {
    __shared__ int cnt[RS_WARPS][256];
    __shared__ int pre[RS_WARPS][256];
    __shared__ int off_s[256];
    __shared__ int wtot[RS_WARPS];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    {
        // thread d: digit d's total and its count in the tiles before this one
        const int d = threadIdx.x;
        const int *row = hcur + (int64_t)d * n_tiles;
        int tot = 0, before = 0;
#pragma unroll 16
        for (int t = 0; t < n_tiles; ++t) {
            const int c = row[t];
            tot += c;
            before += t < (int)blockIdx.x ? c : 0;
        }
        int incl = tot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int x = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += x;
        }
        if (lane == 31) wtot[warp] = incl;
        __syncthreads();
        int wpre = 0;
        for (int w = 0; w < warp; ++w) wpre += wtot[w];
        off_s[d] = wpre + incl - tot + before;
        if (hzero) hzero[(int64_t)d * n_tiles + blockIdx.x] = 0;
    }
    const int64_t base =
        (int64_t)blockIdx.x * RS_SMALL_TILE + (int64_t)warp * (32 * RS_SMALL_ITEMS);
    uint32_t k[RS_SMALL_ITEMS], v[RS_SMALL_ITEMS];
    int loc[RS_SMALL_ITEMS];
    rs_rank<RS_SMALL_ITEMS>(keys, vals, n, base, shift, mask, k, v, loc, cnt, pre);   // syncs the CTA
#pragma unroll
    for (int r = 0; r < RS_SMALL_ITEMS; ++r) {
        const int64_t idx = base + r * 32 + lane;
        const bool ok = idx < n;
        const uint32_t d = (k[r] >> shift) & mask;
        const int pos = ok ? off_s[d] + pre[warp][d] + loc[r] : 0;
        if (ok) {
            okeys[pos] = k[r];
            ovals[pos] = v[r];
        }
        if (hnext) {
            // one atomic per distinct (next digit, destination tile) of the
            // warp's round: a high digit has few values, whose counters
            // would otherwise take the whole round's atomics each
            const uint32_t slot =
                ok ? ((k[r] >> shift_next) & mask_next) * (uint32_t)n_tiles +
                         (uint32_t)(pos / RS_SMALL_TILE)
                   : 0xffffffffu;
            const unsigned peers = __match_any_sync(0xffffffffu, slot);
            if (ok && lane == __ffs(peers) - 1) atomicAdd(&hnext[slot], (int)__popc(peers));
        }
    }
}

size_t radix_tmp_bytes(int64_t n) {
    int64_t n_tiles = ceil_div<int64_t>(n, RS_TILE);
    int64_t m = 256 * n_tiles;
    const size_t big = (size_t)(2 * m + 1) * sizeof(int64_t) + scan_tmp_bytes(m) + 256;
    const int64_t st = ceil_div<int64_t>(n, RS_SMALL_TILE);
    const size_t small = st <= RS_SMALL_TILES ? (size_t)3 * 256 * st * sizeof(int) + 256 : 0;
    return big > small ? big : small;
}

cudaError_t radix_sort_pairs(uint32_t *keys, uint32_t *vals, uint32_t *keys_alt,
                             uint32_t *vals_alt, int64_t n, int bits, void *tmp,
                             size_t tmp_bytes, cudaStream_t st, bool *result_in_alt,
                             int *launches) {
    *result_in_alt = false;
    if (n <= 1 || bits <= 0) return cudaSuccess;
    if (tmp_bytes < radix_tmp_bytes(n)) return cudaErrorInvalidValue;
    const int64_t n_tiles = ceil_div<int64_t>(n, RS_TILE);
    const int64_t m = 256 * n_tiles;
    int64_t *hist = (int64_t *)tmp;
    int64_t *offs = hist + m;
    void *stmp = (void *)(offs + m + 1);
    size_t stmp_bytes = tmp_bytes - (size_t)(2 * m + 1) * sizeof(int64_t);
    uint32_t *ki = keys, *vi = vals, *ko = keys_alt, *vo = vals_alt;
    const int64_t s_tiles = ceil_div<int64_t>(n, RS_SMALL_TILE);
    if (s_tiles <= RS_SMALL_TILES) {
        const int64_t ms = 256 * s_tiles;
        int *h[3] = {(int *)tmp, (int *)tmp + ms, (int *)tmp + 2 * ms};
        const int nt = (int)s_tiles;
        k_rs_hist32<<<nt, RS_THREADS, 0, st>>>(ki, n, 0, bits < 8 ? (1u << bits) - 1u : 0xffu, nt,
                                               h[0], h[1], h[2]);
        if (launches) *launches += 1;
        for (int p = 0, sh = 0; sh < bits; ++p, sh += 8) {
            const int nb = bits - sh < 8 ? bits - sh : 8;
            const int shn = sh + 8;
            const int nbn = bits - shn < 8 ? bits - shn : 8;
            k_rs_scatter_small<<<nt, RS_THREADS, 0, st>>>(
                ki, vi, n, sh, (1u << nb) - 1u, nt, h[p % 3], shn < bits ? h[(p + 1) % 3] : nullptr,
                shn, shn < bits ? (1u << nbn) - 1u : 0u, p >= 1 ? h[(p + 2) % 3] : nullptr, ko, vo);
            if (launches) *launches += 1;
            cudaError_t e = cudaGetLastError();
            if (e != cudaSuccess) return e;
            uint32_t *t;
            t = ki; ki = ko; ko = t;
            t = vi; vi = vo; vo = t;
            *result_in_alt = !*result_in_alt;
        }
        return cudaSuccess;
    }
    for (int sh = 0; sh < bits; sh += 8) {
        int nb = bits - sh < 8 ? bits - sh : 8;
        uint32_t mask = (1u << nb) - 1u;
        k_rs_hist<<<(unsigned)n_tiles, RS_THREADS, 0, st>>>(ki, n, sh, mask, n_tiles, hist);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        e = scan_exclusive(hist, offs, m, stmp, stmp_bytes, st, launches);
        if (e != cudaSuccess) return e;
        k_rs_scatter<<<(unsigned)n_tiles, RS_THREADS, 0, st>>>(ki, vi, n, sh, mask, n_tiles, offs,
                                                                ko, vo);
        if (launches) *launches += 2;
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        uint32_t *t;
        t = ki; ki = ko; ko = t;
        t = vi; vi = vo; vo = t;
        *result_in_alt = !*result_in_alt;
    }
    return cudaSuccess;
}

// ================================================================== CSR helpers
// One warp per row: src[e] = global row id for every edge of the row, and the
// row is checked: targets in [0, n_total), never the row itself, strictly
// ascending.  row_ptr is relative (offsets into col), rows are local; the
// global id of local row r is row_base + r; edge e is written at out_off + e.
__global__ void k_edge_src_check(const int64_t *__restrict__ row_ptr, const int32_t *__restrict__ col,
                                 int64_t n_rows, int64_t row_base, int64_t n_total,
                                 int32_t *__restrict__ src, int *status) {
    const int lane = threadIdx.x & 31;
    int64_t r = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t stride = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t p0 = row_ptr[0];
    for (; r < n_rows; r += stride) {
        int64_t a = row_ptr[r], b = row_ptr[r + 1];
        if (b < a) {
            if (lane == 0) set_status(status, AKASHIC_EDEVICE);
            continue;
        }
        const int64_t gid = row_base + r;
        for (int64_t e = a + lane; e < b; e += 32) {
            int32_t c = col[e];
            bool bad = c < 0 || (int64_t)c >= n_total || (int64_t)c == gid ||
                       (e > a && col[e - 1] >= c);
            if (bad) set_status(status, AKASHIC_EDEVICE);
            if (src) src[e - p0] = (int32_t)gid;
        }
    }
}

cudaError_t launch_edge_src_check(const int64_t *row_ptr, const int32_t *col, int64_t n_rows,
                                  int64_t row_base, int64_t n_total, int32_t *src, int *status,
                                  cudaStream_t st) {
    if (n_rows <= 0) return cudaSuccess;
    int64_t warps = n_rows < (int64_t)device_sm_count() * 64 ? n_rows : (int64_t)device_sm_count() * 64;
    k_edge_src_check<<<(unsigned)ceil_div<int64_t>(warps * 32, 256), 256, 0, st>>>(
        row_ptr, col, n_rows, row_base, n_total, src, status);
    return cudaGetLastError();
}

// Relation weights: w = softmax of each row's edge logits.  Eight lanes per
// row and four rows per warp step (rows are short: 32 edges plus the
// reciprocal ones), so a warp keeps four rows' loads in flight; a row of up
// to 64 edges is read once and kept in registers.
constexpr int RSM_LANES = 8, RSM_KEEP = 8;
__global__ void k_row_softmax(const int64_t *__restrict__ row_ptr, const float *__restrict__ aff,
                              float *__restrict__ w, int64_t n_rows, float2 *__restrict__ rstat) {
    constexpr int L = RSM_LANES, R = 32 / RSM_LANES;
    const int lane = threadIdx.x & 31, sub = lane % L, grp = lane / L;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    // the next step's row bounds are loaded while this step's rows are
    // processed (they head each step's chain of dependent loads)
    int64_t r0 = (((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5) * R;
    int64_t na = 0, nb = 0;
    if (r0 + grp < n_rows) {
        na = row_ptr[r0 + grp];
        nb = row_ptr[r0 + grp + 1];
    }
    for (; r0 < n_rows; r0 += nw * R) {
        const int64_t r = r0 + grp;
        const int64_t a = na, b = nb;
        const int64_t rn = r + nw * R;
        na = rn < n_rows ? row_ptr[rn] : 0;
        nb = rn < n_rows ? row_ptr[rn + 1] : 0;
        float v[RSM_KEEP];
        float m = -INFINITY;
#pragma unroll
        for (int t = 0; t < RSM_KEEP; ++t) {
            const int64_t e = a + sub + t * L;
            v[t] = e < b ? aff[e] : -INFINITY;
            m = fmaxf(m, v[t]);
        }
        for (int64_t e = a + sub + RSM_KEEP * L; e < b; e += L) m = fmaxf(m, aff[e]);
#pragma unroll
        for (int o = L / 2; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        float s = 0.f;
#pragma unroll
        for (int t = 0; t < RSM_KEEP; ++t)
            if (a + sub + t * L < b) s += expf(v[t] - m);
        for (int64_t e = a + sub + RSM_KEEP * L; e < b; e += L) s += expf(aff[e] - m);
#pragma unroll
        for (int o = L / 2; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (b > a) {
            const float2 stat = make_float2(m, 1.f / s);
            if (rstat && sub == 0) rstat[r] = stat;
#pragma unroll
            for (int t = 0; t < RSM_KEEP; ++t) {
                const int64_t e = a + sub + t * L;
                if (e < b) w[e] = row_softmax_weight(v[t], stat);
            }
            for (int64_t e = a + sub + RSM_KEEP * L; e < b; e += L)
                w[e] = row_softmax_weight(aff[e], stat);
        }
    }
}

cudaError_t launch_row_softmax(const int64_t *row_ptr, const float *aff, float *w, int64_t n_rows,
                               float2 *rstat, cudaStream_t st) {
    if (n_rows <= 0) return cudaSuccess;
    const int64_t want = ceil_div<int64_t>(n_rows, 32 / RSM_LANES);
    const int64_t warps = want < (int64_t)device_sm_count() * 64 ? want : (int64_t)device_sm_count() * 64;
    k_row_softmax<<<(unsigned)ceil_div<int64_t>(warps * 32, 256), 256, 0, st>>>(row_ptr, aff, w,
                                                                              n_rows, rstat);
    return cudaGetLastError();
}

// In-degree of every store row (targets mapped from chunk IDs to rows).
__global__ void k_in_degree(const int32_t *__restrict__ col, const int32_t *__restrict__ row_of,
                            int64_t nnz, unsigned long long *__restrict__ deg) {
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < nnz;
         e += (int64_t)gridDim.x * blockDim.x)
        atomicAdd(&deg[row_of[col[e]]], 1ull);
}

cudaError_t launch_in_degree(const int32_t *col, const int32_t *row_of, int64_t nnz, int64_t *deg,
                             cudaStream_t st) {
    if (nnz <= 0) return cudaSuccess;
    int grid = (int)(nnz / 256 + 1 < (int64_t)device_sm_count() * 16 ? nnz / 256 + 1
                                                                     : device_sm_count() * 16);
    k_in_degree<<<grid, 256, 0, st>>>(col, row_of, nnz, (unsigned long long *)deg);
    return cudaGetLastError();
}

// keys[i] = row_of[ids[sel ? sel[i] : i]]: chunk IDs (of edge sources or
// targets) mapped to store rows, optionally through a permutation.
__global__ void k_map_keys(const uint32_t *__restrict__ sel, const int32_t *__restrict__ ids,
                           const int32_t *__restrict__ row_of, uint32_t *__restrict__ keys,
                           int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        keys[i] = (uint32_t)row_of[ids[sel ? sel[i] : (uint32_t)i]];
}

cudaError_t launch_map_keys(const uint32_t *sel, const int32_t *ids, const int32_t *row_of,
                            uint32_t *keys, int64_t n, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_map_keys<<<device_sm_count() * 8, 256, 0, st>>>(sel, ids, row_of, keys, n);
    return cudaGetLastError();
}

__global__ void k_iota_u32(uint32_t *__restrict__ v, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        v[i] = (uint32_t)i;
}

cudaError_t launch_iota(uint32_t *v, int64_t n, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_iota_u32<<<device_sm_count() * 8, 256, 0, st>>>(v, n);
    return cudaGetLastError();
}

__global__ void k_gather_in(const uint32_t *__restrict__ order, const int32_t *__restrict__ src,
                            const int32_t *__restrict__ row_of, const float *__restrict__ w,
                            const float *__restrict__ aff, int32_t *__restrict__ in_src,
                            float *__restrict__ in_w, float *__restrict__ in_aff, int64_t nnz) {
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < nnz;
         p += (int64_t)gridDim.x * blockDim.x) {
        uint32_t e = order[p];
        in_src[p] = row_of[src[e]];
        in_w[p] = w[e];
        in_aff[p] = aff[e];
    }
}

cudaError_t launch_gather_in(const uint32_t *order, const int32_t *src, const int32_t *row_of,
                             const float *w, const float *aff, int32_t *in_src, float *in_w,
                             float *in_aff, int64_t nnz, cudaStream_t st) {
    if (nnz <= 0) return cudaSuccess;
    k_gather_in<<<device_sm_count() * 8, 256, 0, st>>>(order, src, row_of, w, aff, in_src, in_w,
                                                       in_aff, nnz);
    return cudaGetLastError();
}

// Lay out one append batch in page order: row first+i of the store takes
// chunk first+order[i] (embedding row, page, ID maps).  One warp per row.
__global__ void k_batch_layout(const uint32_t *__restrict__ order, int64_t first, int64_t n,
                               int dim, const uint16_t *__restrict__ emb_in,
                               uint16_t *__restrict__ emb, const int32_t *__restrict__ page_in,
                               int64_t first_page, int per_page, int32_t *__restrict__ page_row,
                               int32_t *__restrict__ ext_of, int32_t *__restrict__ row_of) {
    const int lane = threadIdx.x & 31;
    int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t stride = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int words = dim / 8;   // 16-byte words per row (dim is a multiple of 64)
    for (; i < n; i += stride) {
        const int64_t o = order ? (int64_t)order[i] : i;
        const uint4 *src = (const uint4 *)(emb_in + o * dim);
        uint4 *dst = (uint4 *)(emb + (first + i) * dim);
        for (int t = lane; t < words; t += 32) dst[t] = src[t];
        if (lane == 0) {
            ext_of[first + i] = (int32_t)(first + o);
            row_of[first + o] = (int32_t)(first + i);
            page_row[first + i] = page_in ? page_in[o] : (int32_t)(first_page + o / per_page);
        }
    }
}

cudaError_t launch_batch_layout(const uint32_t *order, int64_t first, int64_t n, int dim,
                                const uint16_t *emb_in, uint16_t *emb, const int32_t *page_in,
                                int64_t first_page, int per_page, int32_t *page_row,
                                int32_t *ext_of, int32_t *row_of, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_batch_layout<<<device_sm_count() * 8, 256, 0, st>>>(order, first, n, dim, emb_in, emb,
                                                          page_in, first_page, per_page, page_row,
                                                          ext_of, row_of);
    return cudaGetLastError();
}

// out[row_of[first + i]] = in[i] for i < n (per-chunk values into row order).
__global__ void k_scatter_by_row(const int32_t *__restrict__ in, const int32_t *__restrict__ row_of,
                                 int64_t first, int64_t n, int32_t *__restrict__ out) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        out[row_of[first + i]] = in[i];
}

cudaError_t launch_scatter_by_row(const int32_t *in, const int32_t *row_of, int64_t first,
                                  int64_t n, int32_t *out, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_scatter_by_row<<<device_sm_count() * 2, 256, 0, st>>>(in, row_of, first, n, out);
    return cudaGetLastError();
}

// Split plan.  A row with more than SPLIT_T in-edges is cut at every source
// window boundary (sources are sorted within a row, so the cut points are
// found by binary search) and then every SEG_LEN edges.
__device__ __forceinline__ int64_t lower_bound_src(const int32_t *__restrict__ src, int64_t lo,
                                                   int64_t hi, int64_t key) {
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if ((int64_t)src[mid] < key) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

// A hub row (more than split_t in-edges, sorted by source row) cut by one
// warp: lane l takes source windows w0 + l, w0 + l + 32, ...; the edge range
// of each window comes from two binary searches, and its segments (at most
// seg_len edges each) are numbered by a scan across the lanes in window
// order.  Returns the row's segment count (on every lane).
template <bool FILL>
__device__ int64_t warp_segments(const SplitParams &sp, const int32_t *__restrict__ in_src,
                                 int64_t a, int64_t b, int64_t slot, int64_t *seg_e0,
                                 int64_t *seg_e1, uint32_t *seg_win) {
    const int lane = threadIdx.x & 31;
    const int64_t w0 = (int64_t)in_src[a] / sp.win_rows, w1 = (int64_t)in_src[b - 1] / sp.win_rows;
    int64_t base = 0;
    for (int64_t wb = w0; wb <= w1; wb += 32) {
        const int64_t w = wb + lane;
        int64_t lo = 0, cnt = 0, hi = 0;
        if (w <= w1) {
            lo = w == w0 ? a : lower_bound_src(in_src, a, b, w * sp.win_rows);
            hi = w == w1 ? b : lower_bound_src(in_src, lo, b, (w + 1) * sp.win_rows);
            cnt = (hi - lo + sp.seg_len - 1) / sp.seg_len;
        }
        int64_t incl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int64_t t = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += t;
        }
        if (FILL) {
            const int64_t at = slot + base + incl - cnt;
            for (int64_t t = 0; t < cnt; ++t) {
                const int64_t e = lo + t * sp.seg_len;
                seg_e0[at + t] = e;
                seg_e1[at + t] = e + sp.seg_len < hi ? e + sp.seg_len : hi;
                seg_win[at + t] = (uint32_t)w;
            }
        }
        base += __shfl_sync(0xffffffffu, incl, 31);
    }
    return base;
}

// Segment count of every row (0 below split_t).  A warp takes 32 rows; its
// hub rows are then cut one after another by the whole warp.
__global__ void k_split_count(SplitParams sp, const int64_t *__restrict__ in_ptr,
                              const int32_t *__restrict__ in_src, int64_t n,
                              int64_t *__restrict__ nseg, int64_t *__restrict__ flag) {
    const int lane = threadIdx.x & 31;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t r0 = (((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5) * 32; r0 < n;
         r0 += nw * 32) {
        const int64_t j = r0 + lane;
        bool heavy = false;
        if (j < n) {
            heavy = in_ptr[j + 1] - in_ptr[j] > sp.split_t;
            if (!heavy) {
                nseg[j] = 0;
                flag[j] = 0;
            }
        }
        unsigned hv = __ballot_sync(0xffffffffu, heavy);
        while (hv) {
            const int l = __ffs(hv) - 1;
            hv &= hv - 1;
            const int64_t h = r0 + l;
            const int64_t s = warp_segments<false>(sp, in_src, in_ptr[h], in_ptr[h + 1], 0, nullptr,
                                                   nullptr, nullptr);
            if (lane == 0) {
                nseg[h] = s;
                flag[h] = s > 0;
            }
        }
    }
}

__global__ void k_split_fill(SplitParams sp, const int64_t *__restrict__ in_ptr,
                             const int32_t *__restrict__ in_src, int64_t n,
                             const int64_t *__restrict__ nseg,
                             const int64_t *__restrict__ slot_off,
                             const int64_t *__restrict__ split_idx, int32_t *__restrict__ split_row,
                             int64_t *__restrict__ split_slot0, int64_t *__restrict__ seg_e0,
                             int64_t *__restrict__ seg_e1, uint32_t *__restrict__ seg_win) {
    const int lane = threadIdx.x & 31;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t r0 = (((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5) * 32; r0 < n;
         r0 += nw * 32) {
        const int64_t j = r0 + lane;
        unsigned hv = __ballot_sync(0xffffffffu, j < n && nseg[j] > 0);
        while (hv) {
            const int l = __ffs(hv) - 1;
            hv &= hv - 1;
            const int64_t h = r0 + l;
            if (lane == 0) {
                const int64_t idx = split_idx[h];
                split_row[idx] = (int32_t)h;
                split_slot0[idx] = slot_off[h];
            }
            warp_segments<true>(sp, in_src, in_ptr[h], in_ptr[h + 1], slot_off[h], seg_e0, seg_e1,
                                seg_win);
        }
    }
}

__global__ void k_seg_permute(const uint32_t *__restrict__ order, const int64_t *__restrict__ e0,
                              const int64_t *__restrict__ e1, int64_t n_segs,
                              int64_t *__restrict__ e0s, int64_t *__restrict__ e1s,
                              int32_t *__restrict__ slot) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n_segs;
         i += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t o = order[i];
        e0s[i] = e0[o];
        e1s[i] = e1[o];
        slot[i] = (int32_t)o;
    }
}

cudaError_t launch_split_count(const SplitParams &sp, const int64_t *in_ptr, const int32_t *in_src,
                               int64_t n, int64_t *nseg, int64_t *flag, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_split_count<<<device_sm_count() * 4, 256, 0, st>>>(sp, in_ptr, in_src, n, nseg, flag);
    return cudaGetLastError();
}

cudaError_t launch_split_fill(const SplitParams &sp, const int64_t *in_ptr, const int32_t *in_src,
                              int64_t n, const int64_t *nseg, const int64_t *slot_off,
                              const int64_t *split_idx, int32_t *split_row, int64_t *split_slot0,
                              int64_t *seg_e0, int64_t *seg_e1, uint32_t *seg_win,
                              cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_split_fill<<<device_sm_count() * 4, 256, 0, st>>>(sp, in_ptr, in_src, n, nseg, slot_off,
                                                        split_idx, split_row, split_slot0, seg_e0,
                                                        seg_e1, seg_win);
    return cudaGetLastError();
}

cudaError_t launch_seg_permute(const uint32_t *order, const int64_t *e0, const int64_t *e1,
                               int64_t n_segs, int64_t *e0s, int64_t *e1s, int32_t *slot,
                               cudaStream_t st) {
    if (n_segs <= 0) return cudaSuccess;
    k_seg_permute<<<device_sm_count() * 2, 256, 0, st>>>(order, e0, e1, n_segs, e0s, e1s, slot);
    return cudaGetLastError();
}

// Split rows ordered by their number of partial slots, largest first (the
// hop sums each split row's slots in one warp and hands the heaviest out
// first, so that they finish early).  keys = ~count, so an ascending stable
// sort gives descending counts with ties in row order.
__global__ void k_split_keys(const int64_t *__restrict__ slot0, int64_t n_split,
                             uint32_t *__restrict__ keys, uint32_t *__restrict__ vals) {
    for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n_split;
         r += (int64_t)gridDim.x * blockDim.x) {
        keys[r] = ~(uint32_t)(slot0[r + 1] - slot0[r]);
        vals[r] = (uint32_t)r;
    }
}

cudaError_t launch_split_keys(const int64_t *slot0, int64_t n_split, uint32_t *keys,
                              uint32_t *vals, cudaStream_t st) {
    if (n_split <= 0) return cudaSuccess;
    k_split_keys<<<device_sm_count(), 256, 0, st>>>(slot0, n_split, keys, vals);
    return cudaGetLastError();
}

// ================================================================== propagation hop
// out[j,:] = u[j,:] + alpha * sum_{i->j} w_ij in[i,:], gathered over the
// in-edge CSR, one warp per destination row.  A row holds BP fp32 values
// (BP/4 float4).  For BP >= 128 each lane owns BP/128 float4 of the row; for
// smaller BP the warp splits into 32/(BP/4) lane groups that take
// alternate edges and are summed at the end.  Rows with more than split_t
// in-edges are skipped here and handled by window segments + fixup.
// L2 policy for the hop: gathered source rows are re-read ~32 times (once
// per out-edge of the source), so they are loaded with an evict-last
// policy; everything read or written once (graph arrays, u, the output
// slab, partial sums) streams with evict-first (.cs) accesses so that it
// does not push gathered rows out of L2.
__device__ __forceinline__ uint64_t l2_keep_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ float4 ld_keep(const float4 *p, uint64_t pol) {
    float4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.f32 {%0,%1,%2,%3}, [%4], %5;"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p), "l"(pol));
    return v;
}
__device__ __forceinline__ float4 ld_stream(const float4 *p) { return __ldcs(p); }
__device__ __forceinline__ void st_stream(float4 *p, float4 v) { __stcs(p, v); }
__device__ __forceinline__ int32_t ld_stream(const int32_t *p) { return __ldcs(p); }
__device__ __forceinline__ float ld_stream(const float *p) { return __ldcs(p); }

template <int BP>
struct HopShape {
    static constexpr int F = BP / 4;                       // float4 per row
    static constexpr int G = F >= 32 ? 1 : 32 / F;         // edge groups per warp
    static constexpr int V = F >= 32 ? F / 32 : 1;         // float4 per lane
    static constexpr int LW = F >= 32 ? 32 : F;            // lanes per group
};

template <int BP, int WIDTH = 1>
__device__ __forceinline__ void hop_accumulate(const int32_t *__restrict__ in_src,
                                               const float *__restrict__ in_w, int64_t e0,
                                               int64_t e1, const float4 *__restrict__ in4,
                                               float4 (&acc)[HopShape<BP>::V]) {
    using S = HopShape<BP>;
    // gathers in flight: UN edges x V float4 (WIDTH times more in the wide
    // variant, which runs fewer warps)
    constexpr int UN = WIDTH * (8 / S::V > 0 ? 8 / S::V : 1);
    const int lane = threadIdx.x & 31;
    const int g = lane / S::LW, sub = lane % S::LW;
    const uint64_t pol = l2_keep_policy();
#pragma unroll
    for (int v = 0; v < S::V; ++v) acc[v] = make_float4(0.f, 0.f, 0.f, 0.f);
    // the next batch's (source, weight) pairs are loaded while this batch gathers
    int32_t s_n = 0;
    float w_n = 0.f;
    if (e0 + lane < e1) {
        s_n = ld_stream(in_src + e0 + lane);
        w_n = ld_stream(in_w + e0 + lane);
    }
    for (int64_t eb = e0; eb < e1; eb += 32) {
        const int cnt = (int)(e1 - eb < 32 ? e1 - eb : 32);
        const int32_t s_l = s_n;
        const float w_l = w_n;
        if (eb + 32 + lane < e1) {
            s_n = ld_stream(in_src + eb + 32 + lane);
            w_n = ld_stream(in_w + eb + 32 + lane);
        }
        int t = 0;
        for (; t + UN * S::G <= cnt; t += UN * S::G) {
            int32_t sq[UN];
            float wq[UN];
#pragma unroll
            for (int q = 0; q < UN; ++q) {
                sq[q] = __shfl_sync(0xffffffffu, s_l, t + q * S::G + g);
                wq[q] = __shfl_sync(0xffffffffu, w_l, t + q * S::G + g);
            }
            float4 x[UN][S::V];
#pragma unroll
            for (int q = 0; q < UN; ++q)
#pragma unroll
                for (int v = 0; v < S::V; ++v)
                    x[q][v] = ld_keep(in4 + (int64_t)sq[q] * S::F + sub + 32 * v, pol);
#pragma unroll
            for (int q = 0; q < UN; ++q)
#pragma unroll
                for (int v = 0; v < S::V; ++v) {
                    acc[v].x = fmaf(wq[q], x[q][v].x, acc[v].x);
                    acc[v].y = fmaf(wq[q], x[q][v].y, acc[v].y);
                    acc[v].z = fmaf(wq[q], x[q][v].z, acc[v].z);
                    acc[v].w = fmaf(wq[q], x[q][v].w, acc[v].w);
                }
        }
        for (; t < cnt; t += S::G) {
            const int idx = t + g;
            int32_t sv = __shfl_sync(0xffffffffu, s_l, idx < 32 ? idx : 31);
            float wv = __shfl_sync(0xffffffffu, w_l, idx < 32 ? idx : 31);
            if (idx < cnt) {
#pragma unroll
                for (int v = 0; v < S::V; ++v) {
                    float4 x = ld_keep(in4 + (int64_t)sv * S::F + sub + 32 * v, pol);
                    acc[v].x = fmaf(wv, x.x, acc[v].x);
                    acc[v].y = fmaf(wv, x.y, acc[v].y);
                    acc[v].z = fmaf(wv, x.z, acc[v].z);
                    acc[v].w = fmaf(wv, x.w, acc[v].w);
                }
            }
        }
    }
    if (S::G > 1) {
#pragma unroll
        for (int o = S::LW; o < 32; o <<= 1) {
#pragma unroll
            for (int v = 0; v < S::V; ++v) {
                acc[v].x += __shfl_xor_sync(0xffffffffu, acc[v].x, o);
                acc[v].y += __shfl_xor_sync(0xffffffffu, acc[v].y, o);
                acc[v].z += __shfl_xor_sync(0xffffffffu, acc[v].z, o);
                acc[v].w += __shfl_xor_sync(0xffffffffu, acc[v].w, o);
            }
        }
    }
}

// ------------------------------------------------------------------ row bounds
// Scalar bounds on the hops' fp32 values, one pair per row: U[j] is at least
// and L[j] at most every real query column's value of s^(h)_j.  Level 0 is
// u's row maximum / minimum (from the score step); level h follows the hop
// s^(h)_j = fma(alpha, sum_{i->j} w_ij s^(h-1)_i, u_j) with the sums of
// w * U and w * L over the row's in-edges (w, s >= 0), widened for rounding:
// the hop's sum takes at most 2n + 10 roundings on any term's path
// (segments and partial slots included) and the bound's own sum at most
// n + 5, so exp(+-x), x = 3.25 (n + 8) 2^-24, covers both (with 1 + x + x^2
// >= exp(x) and 1 - x <= exp(-x) for 0 <= x <= 1), and a factor 1 -+ 4e-6
// (~67 ulp) covers the final rounding of the hop and of evaluating the
// bound in fp32.
__device__ __forceinline__ float bound_x(int64_t n) {
    return 3.25f * (float)(n + 8) * 5.9604645e-8f;
}
__device__ __forceinline__ float bound_up(float u0, float v, int64_t n, float alpha) {
    const float x = bound_x(n);
    if (!(x <= 1.f)) return INFINITY;
    return fmaf(alpha * v, 1.f + x + x * x, u0) * (1.f + 4e-6f);
}
__device__ __forceinline__ float bound_dn(float l0, float v, int64_t n, float alpha) {
    const float x = bound_x(n);
    const float g = x < 1.f ? 1.f - x : 0.f;
    return fmaf(alpha * v, g, l0) * (1.f - 4e-6f);
}

// The sums of w * U[source] and w * L[source] over in-edges e0..e1, by a
// group of LN lanes (lane `sl` of the group), four edges in flight per lane;
// every lane of the group returns them.
template <int LN>
__device__ __forceinline__ void bound_sums(const int32_t *__restrict__ in_src,
                                           const float *__restrict__ in_w, int64_t e0, int64_t e1,
                                           const float *__restrict__ U, const float *__restrict__ L,
                                           int sl, float &vu, float &vl) {
    vu = 0.f;
    vl = 0.f;
    for (int64_t eb = e0 + sl; eb < e1; eb += 4 * LN) {
        int32_t s[4];
        float w[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int64_t e = eb + LN * q;
            s[q] = e < e1 ? __ldcs(in_src + e) : 0;
            w[q] = e < e1 ? __ldcs(in_w + e) : 0.f;
        }
        float a[4], c[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const bool in = eb + LN * q < e1;
            a[q] = in ? __ldg(U + s[q]) : 0.f;
            c[q] = in ? __ldg(L + s[q]) : 0.f;
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            vu = fmaf(w[q], a[q], vu);
            vl = fmaf(w[q], c[q], vl);
        }
    }
#pragma unroll
    for (int off = LN / 2; off > 0; off >>= 1) {
        vu += __shfl_xor_sync(0xffffffffu, vu, off);
        vl += __shfl_xor_sync(0xffffffffu, vl, off);
    }
}

// One level for the rows kept whole: four lanes per row, eight rows per warp.
constexpr int BND_LANES = 4;
__global__ void k_bound_rows(const int64_t *__restrict__ in_ptr, const int32_t *__restrict__ in_src,
                             const float *__restrict__ in_w, int64_t n, int64_t split_t,
                             const float *__restrict__ u0, const float *__restrict__ l0,
                             const float *__restrict__ Up, const float *__restrict__ Lp,
                             float alpha, float *__restrict__ Un, float *__restrict__ Ln) {
    constexpr int R = 32 / BND_LANES;
    const int lane = threadIdx.x & 31, sl = lane % BND_LANES, grp = lane / BND_LANES;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t r0 = (((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5) * R; r0 < n;
         r0 += nw * R) {
        const int64_t j = r0 + grp;
        int64_t e0 = 0, e1 = 0;
        if (j < n) {
            e0 = in_ptr[j];
            e1 = in_ptr[j + 1];
        }
        const bool whole = j < n && e1 - e0 <= split_t;
        float vu, vl;
        bound_sums<BND_LANES>(in_src, in_w, e0, whole ? e1 : e0, Up, Lp, sl, vu, vl);
        if (whole && sl == 0) {
            Un[j] = bound_up(u0[j], vu, e1 - e0, alpha);
            Ln[j] = bound_dn(l0[j], vl, e1 - e0, alpha);
        }
    }
}

// Split rows: one warp per segment, its sums added into the owning row's
// totals (the order of the additions does not change the bound: every
// term is >= 0 and a term's path stays within the row's edge count + 5
// roundings) ...
__global__ void k_seg_bound(const int64_t *__restrict__ seg_e0, const int64_t *__restrict__ seg_e1,
                            const int32_t *__restrict__ seg_slot, int64_t n_segs,
                            const int32_t *__restrict__ slot_split,
                            const int32_t *__restrict__ in_src, const float *__restrict__ in_w,
                            const float *__restrict__ Up, const float *__restrict__ Lp,
                            float *__restrict__ split_vu, float *__restrict__ split_vl) {
    const int lane = threadIdx.x & 31;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t s = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; s < n_segs; s += nw) {
        float vu, vl;
        bound_sums<32>(in_src, in_w, seg_e0[s], seg_e1[s], Up, Lp, lane, vu, vl);
        if (lane == 0) {
            const int32_t r = slot_split[seg_slot[s]];
            atomicAdd(split_vu + r, vu);
            atomicAdd(split_vl + r, vl);
        }
    }
}

// ... then each split row's bounds.
__global__ void k_split_bound(const int64_t *__restrict__ in_ptr, int64_t n_split,
                              const int32_t *__restrict__ split_row,
                              const float *__restrict__ u0, const float *__restrict__ l0,
                              const float *__restrict__ split_vu, const float *__restrict__ split_vl,
                              float alpha, float *__restrict__ Un, float *__restrict__ Ln) {
    for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n_split;
         r += (int64_t)gridDim.x * blockDim.x) {
        const int64_t j = split_row[r];
        const int64_t n = in_ptr[j + 1] - in_ptr[j];
        Un[j] = bound_up(u0[j], split_vu[r], n, alpha);
        Ln[j] = bound_dn(l0[j], split_vl[r], n, alpha);
    }
}

// Last hop: split rows whose bound stays below the floor, and their partial
// slots (the segment kernel skips those).  One warp per row.
__global__ void k_split_flags(int64_t n_split, const int32_t *__restrict__ split_row,
                              const int64_t *__restrict__ split_slot0,
                              const float *__restrict__ row_ub, const float *__restrict__ floor_p,
                              const NsFloors nf, int32_t *__restrict__ split_skip,
                              int32_t *__restrict__ slot_skip) {
    const float floor_ = *floor_p;
    const int lane = threadIdx.x & 31;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t r = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < n_split; r += nw) {
        const int32_t j = split_row[r];
        const int32_t skip = row_ub[j] < row_floor(nf, floor_, j) ? 1 : 0;
        if (lane == 0) split_skip[r] = skip;
        for (int64_t s = split_slot0[r] + lane; s < split_slot0[r + 1]; s += 32) slot_skip[s] = skip;
    }
}

__global__ void k_slot_owner(const int64_t *__restrict__ split_slot0, int64_t n_split,
                             int32_t *__restrict__ slot_split) {
    const int lane = threadIdx.x & 31;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t r = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < n_split; r += nw)
        for (int64_t s = split_slot0[r] + lane; s < split_slot0[r + 1]; s += 32)
            slot_split[s] = (int32_t)r;
}

__global__ void k_fill_f32(float *__restrict__ v, int64_t n, float x) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        v[i] = x;
}

cudaError_t launch_fill_f32(float *v, int64_t n, float x, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_fill_f32<<<device_sm_count() * 2, 256, 0, st>>>(v, n, x);
    return cudaGetLastError();
}

cudaError_t launch_slot_owner(const int64_t *split_slot0, int64_t n_split, int32_t *slot_split,
                              cudaStream_t st) {
    if (n_split <= 0) return cudaSuccess;
    k_slot_owner<<<device_sm_count() * 4, 256, 0, st>>>(split_slot0, n_split, slot_split);
    return cudaGetLastError();
}

cudaError_t launch_mass_levels(const HopPlan &p, int t0, int t1, float *mup, float *mdn,
                               const float *zeros, float *split_vu, float *split_vl,
                               cudaStream_t st) {
    const int sms = device_sm_count();
    const int64_t n = p.n;
    for (int t = t0; t <= t1; ++t) {
        const float *Up = mup + (int64_t)(t - 1) * n, *Lp = mdn + (int64_t)(t - 1) * n;
        float *Un = mup + (int64_t)t * n, *Ln = mdn + (int64_t)t * n;
        const int64_t want = ceil_div<int64_t>(n, 32);
        const int g = (int)(want < (int64_t)sms * 8 ? (want < 1 ? 1 : want) : (int64_t)sms * 8);
        k_bound_rows<<<g, 256, 0, st>>>(p.in_ptr, p.in_src, p.in_w, n, p.split.split_t, zeros,
                                         zeros, Up, Lp, 1.f, Un, Ln);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        if (p.n_split_rows > 0) {
            e = cudaMemsetAsync(split_vu, 0, (size_t)p.n_split_rows * 4, st);
            if (e == cudaSuccess) e = cudaMemsetAsync(split_vl, 0, (size_t)p.n_split_rows * 4, st);
            if (e != cudaSuccess) return e;
            const int64_t ws = ceil_div<int64_t>(p.n_segs, 8);
            const int gs = (int)(ws < (int64_t)sms * 8 ? (ws < 1 ? 1 : ws) : (int64_t)sms * 8);
            k_seg_bound<<<gs, 256, 0, st>>>(p.seg_e0, p.seg_e1, p.seg_slot, p.n_segs,
                                            p.slot_split, p.in_src, p.in_w, Up, Lp, split_vu,
                                            split_vl);
            const int64_t wr = ceil_div<int64_t>(p.n_split_rows, 256);
            const int gr = (int)(wr < (int64_t)sms * 2 ? wr : (int64_t)sms * 2);
            k_split_bound<<<gr, 256, 0, st>>>(p.in_ptr, p.n_split_rows, p.split_row, zeros, zeros,
                                              split_vu, split_vl, 1.f, Un, Ln);
            e = cudaGetLastError();
            if (e != cudaSuccess) return e;
        }
    }
    return cudaSuccess;
}

// The store-wide extremes of u's row maxima and (over rows with u > 0, i.e.
// live rows, the only possible edge sources) row minima: ext[0] = Umax,
// ext[1] = Lmin, as float bits (values >= 0 order like their bits).
__global__ void k_row_extremes(const float *__restrict__ u0, const float *__restrict__ l0,
                               int64_t n, unsigned int *__restrict__ ext) {
    unsigned int mx = 0u, mn = 0x7f800000u;
    for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n;
         j += (int64_t)gridDim.x * blockDim.x) {
        const unsigned int a = __float_as_uint(u0[j]);
        mx = a > mx ? a : mx;
        if (a > 0u) {
            const unsigned int b = __float_as_uint(l0[j]);
            mn = b < mn ? b : mn;
        }
    }
    for (int off = 16; off > 0; off >>= 1) {
        const unsigned int x = __shfl_xor_sync(0xffffffffu, mx, off);
        const unsigned int y = __shfl_xor_sync(0xffffffffu, mn, off);
        mx = x > mx ? x : mx;
        mn = y < mn ? y : mn;
    }
    if ((threadIdx.x & 31) == 0) {
        atomicMax(ext, mx);
        atomicMax(ext + 1, 0x7f800000u - mn);
    }
}

// ub_j = (U0_j + Umax * sum_t alpha^t Mup[t]_j) (1 + 1e-5) and
// lb_j = (L0_j + Lmin * sum_t alpha^t Mdn[t]_j) (1 - 1e-5): the (1 +- eps) of
// the hop's last rounding and the at most ~3H roundings of this evaluation
// (Horner, alpha^t) stay far below the 1e-5 (~168 eps) for H <= 16.
__global__ void k_final_bounds(const float *__restrict__ u0, const float *__restrict__ l0,
                               const float *__restrict__ mup, const float *__restrict__ mdn,
                               int64_t n, int H, float alpha, const unsigned int *__restrict__ ext,
                               float *__restrict__ ub, float *__restrict__ lb) {
    const float umax = ext_umax(ext), lmin = ext_lmin(ext);
    for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n;
         j += (int64_t)gridDim.x * blockDim.x) {
        ub[j] = row_upper_bound(u0, mup, n, H, alpha, umax, j);
        lb[j] = row_lower_bound(l0, mdn, n, H, alpha, lmin, j);
    }
}

cudaError_t launch_final_bounds(const float *u0, const float *l0, const float *mup,
                                const float *mdn, int64_t n, int H, float alpha,
                                unsigned int *ext, float *ub, float *lb, cudaStream_t st,
                                int *launches, bool ext_ready) {
    const int sms = device_sm_count();
    if (!ext_ready) {
        cudaError_t e = cudaMemsetAsync(ext, 0, 2 * sizeof(unsigned int), st);
        if (e != cudaSuccess) return e;
        k_row_extremes<<<sms * 4, 256, 0, st>>>(u0, l0, n, ext);
        if (launches) *launches += 1;
    }
    // one row per thread up to 32 CTAs per SM: a few loads per row, so the
    // rows in flight set the rate
    const int64_t fb = ceil_div<int64_t>(n, 256);
    k_final_bounds<<<(unsigned)(fb < (int64_t)sms * 32 ? (fb > 0 ? fb : 1) : (int64_t)sms * 32), 256, 0,
                     st>>>(u0, l0, mup, mdn, n, H, alpha, ext, ub, lb);
    if (launches) *launches += 1;
    return cudaGetLastError();
}

// Last hop: keep flags of the rows kept whole whose bound reaches the floor,
// and of the segments of unpruned split rows; the lists are compacted by an
// exclusive scan, so they keep row order and window-major order (the order
// that keeps gathered source rows in L2).
__global__ void k_keep_rows(const int64_t *__restrict__ in_ptr, int64_t n, int64_t split_t,
                            const float *__restrict__ row_ub, const float *__restrict__ floor_p,
                            const NsFloors nf, int64_t *__restrict__ flag) {
    const float floor_ = *floor_p;
    for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n;
         j += (int64_t)gridDim.x * blockDim.x)
        flag[j] = in_ptr[j + 1] - in_ptr[j] <= split_t && row_ub[j] >= row_floor(nf, floor_, j);
}
__global__ void k_keep_segs(const int32_t *__restrict__ seg_slot, int64_t n_segs,
                            const int32_t *__restrict__ slot_skip, int64_t *__restrict__ flag) {
    for (int64_t s = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; s < n_segs;
         s += (int64_t)gridDim.x * blockDim.x)
        flag[s] = slot_skip[seg_slot[s]] == 0;
}
__global__ void k_compact_kept(const int64_t *__restrict__ flag, const int64_t *__restrict__ pos,
                               int64_t n, int32_t *__restrict__ out, int64_t *__restrict__ count) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        if (flag[i]) out[pos[i]] = (int32_t)i;
    if (blockIdx.x == 0 && threadIdx.x == 0) *count = pos[n];
}

cudaError_t launch_split_flags(const HopPlan &p, const float *row_ub, const float *floor_p,
                               const NsFloors *nf, int32_t *split_skip, int32_t *slot_skip,
                               int32_t *kept_rows, int64_t *kept_count, int32_t *kept_segs,
                               KeptScratch &ks, cudaStream_t st, int *launches) {
    const int sms = device_sm_count();
    const NsFloors f = nf ? *nf : NsFloors{};
    if (p.n_split_rows > 0) {
        const int64_t want = ceil_div<int64_t>(p.n_split_rows, 8);
        const int g = (int)(want < (int64_t)sms * 4 ? want : (int64_t)sms * 4);
        k_split_flags<<<g, 256, 0, st>>>(p.n_split_rows, p.split_row, p.split_slot0, row_ub,
                                         floor_p, f, split_skip, slot_skip);
    }
    if (launches && p.n_split_rows > 0) *launches += 1;
    // kept_count[0]: rows, kept_count[1]: segments
    k_keep_rows<<<sms * 4, 256, 0, st>>>(p.in_ptr, p.n, p.split.split_t, row_ub, floor_p, f,
                                         ks.flag);
    cudaError_t e = scan_exclusive(ks.flag, ks.pos, p.n, ks.tmp, ks.tmp_bytes, st, launches);
    if (e != cudaSuccess) return e;
    k_compact_kept<<<sms * 4, 256, 0, st>>>(ks.flag, ks.pos, p.n, kept_rows, kept_count);
    if (launches) *launches += 2;
    if (p.n_segs > 0) {
        k_keep_segs<<<sms * 4, 256, 0, st>>>(p.seg_slot, p.n_segs, slot_skip, ks.flag);
        e = scan_exclusive(ks.flag, ks.pos, p.n_segs, ks.tmp, ks.tmp_bytes, st, launches);
        if (e != cudaSuccess) return e;
        k_compact_kept<<<sms * 4, 256, 0, st>>>(ks.flag, ks.pos, p.n_segs, kept_segs,
                                                kept_count + 1);
        if (launches) *launches += 2;
    } else {
        e = cudaMemsetAsync(kept_count + 1, 0, sizeof(int64_t), st);
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

// A split row: out = u + alpha * (sum of its partial slots a..b-1), summed
// by one warp in slot order (lane groups take alternate slots and are
// added in group order), so the result does not depend on scheduling.
// Filter epilogue: lane `sub` holds columns (sub + 32 v) * 4 + 0..3 of row j.
// thr[BP] holds the column bounds and thr_hi[BP/4] their upper words (the
// score bits), four columns per uint4 so that a lane's test is one
// conflict-free shared load and four 32-bit compares; only a value whose
// bits reach the bound's (rare: ~ a few k per column) takes the 64-bit
// compare and the append.
template <int BP>
__device__ __noinline__ void hop_filter_row(const HopFilter &f, const unsigned long long *thr,
                                           const uint4 *thr_hi, int sub, int64_t j, uint32_t id,
                                           const float4 (&o)[HopShape<BP>::V]) {
#pragma unroll
    for (int v = 0; v < HopShape<BP>::V; ++v) {
        const uint4 h = thr_hi[sub + 32 * v];
        const uint32_t x[4] = {__float_as_uint(o[v].x), __float_as_uint(o[v].y),
                               __float_as_uint(o[v].z), __float_as_uint(o[v].w)};
        const uint32_t hh[4] = {h.x, h.y, h.z, h.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            if (x[e] >= hh[e]) {
                const int c = (sub + 32 * v) * 4 + e;
                const unsigned long long key =
                    ((unsigned long long)x[e] << 32) | (unsigned long long)(~id);
                if (key >= thr[c] && in_scope(f.ns, j, c)) {
                    const unsigned int p = atomicAdd(&f.cnt[c], 1u);
                    if ((int64_t)p < f.cap) f.buf[(int64_t)c * f.cap + p] = key;
                }
            }
        }
    }
}

// Kept out of line: any inlined test here slowed the whole row loop of the
// hop by ~5% (measured), while a call per row costs ~2%.
template <int BP, bool FILTER>
__device__ __forceinline__ void hop_emit(const HopFilter &f, const unsigned long long *thr,
                                         const uint4 *thr_hi, int sub, int64_t j, uint32_t id,
                                         const float4 (&o)[HopShape<BP>::V]) {
    if constexpr (FILTER) hop_filter_row<BP>(f, thr, thr_hi, sub, j, id, o);
}

template <int BP, bool FILTER, int WIDTH = 1>
__device__ __forceinline__ void hop_fixup_row(int64_t j, int64_t a, int64_t b,
                                              const float4 *__restrict__ part4,
                                              const float4 *__restrict__ u4,
                                              float4 *__restrict__ out4, float alpha,
                                              const HopFilter &f,
                                              const unsigned long long *thr,
                                              const uint4 *thr_hi) {
    using S = HopShape<BP>;
    constexpr int P = WIDTH * (8 / S::V > 0 ? 8 / S::V : 1);   // slots in flight per lane group
    const int lane = threadIdx.x & 31;
    const int g = lane / S::LW, sub = lane % S::LW;
    const uint32_t id = FILTER ? (uint32_t)f.ext_of[j] : 0u;
    float4 acc[S::V];
#pragma unroll
    for (int v = 0; v < S::V; ++v) acc[v] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int64_t t = a; t < b; t += P * S::G) {
        float4 x[P][S::V];
#pragma unroll
        for (int q = 0; q < P; ++q) {
            const int64_t sl = t + q * S::G + g;
#pragma unroll
            for (int v = 0; v < S::V; ++v)
                x[q][v] = sl < b ? ld_stream(part4 + sl * S::F + sub + 32 * v)
                                 : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int q = 0; q < P; ++q)
#pragma unroll
            for (int v = 0; v < S::V; ++v) {
                acc[v].x += x[q][v].x; acc[v].y += x[q][v].y;
                acc[v].z += x[q][v].z; acc[v].w += x[q][v].w;
            }
    }
    if (S::G > 1) {
#pragma unroll
        for (int o = S::LW; o < 32; o <<= 1)
#pragma unroll
            for (int v = 0; v < S::V; ++v) {
                acc[v].x += __shfl_xor_sync(0xffffffffu, acc[v].x, o);
                acc[v].y += __shfl_xor_sync(0xffffffffu, acc[v].y, o);
                acc[v].z += __shfl_xor_sync(0xffffffffu, acc[v].z, o);
                acc[v].w += __shfl_xor_sync(0xffffffffu, acc[v].w, o);
            }
    }
    if (lane < S::LW) {
        float4 o[S::V];
#pragma unroll
        for (int v = 0; v < S::V; ++v) {
            o[v] = ld_stream(u4 + j * S::F + sub + 32 * v);
            o[v].x = fmaf(alpha, acc[v].x, o[v].x);
            o[v].y = fmaf(alpha, acc[v].y, o[v].y);
            o[v].z = fmaf(alpha, acc[v].z, o[v].z);
            o[v].w = fmaf(alpha, acc[v].w, o[v].w);
            if constexpr (!FILTER) st_stream(out4 + j * S::F + sub + 32 * v, o[v]);
        }
        hop_emit<BP, FILTER>(f, thr, thr_hi, sub, j, id, o);
    }
}

// With the filter (the last hop) the output slab is not written: the
// selection needs only the keys the filter appends (a query whose buffer
// overflows gets its column recomputed by the merge).
//
// One queue: first the split rows (their segment partials are complete,
// the segment kernel ran before), heaviest first, one warp each; then the
// rows kept whole, ROWS_PER_GRAB consecutive rows per claim (load
// balance), with the group's row pointers read at once and each row's u
// load issued before its gathers.
// WIDTH 2 (the pruned last hop, few work items): twice the loads in flight
// per warp, two CTAs per SM.
template <int BP, bool FILTER, int WIDTH = 1>
__global__ __launch_bounds__(256, WIDTH > 1 ? 2 : 3) void k_hop_rows(const int64_t *__restrict__ in_ptr,
                                                  const int32_t *__restrict__ in_src,
                                                  const float *__restrict__ in_w, int64_t n,
                                                  const float4 *__restrict__ u4,
                                                  const float4 *__restrict__ in4,
                                                  float4 *__restrict__ out4, float alpha,
                                                  int64_t split_t, int64_t n_split,
                                                  const int32_t *__restrict__ split_order,
                                                  const int32_t *__restrict__ split_row,
                                                  const int64_t *__restrict__ split_slot0,
                                                  const float4 *__restrict__ part4,
                                                  HopFilter f,
                                                  const float *__restrict__ row_ub,
                                                  const float *__restrict__ floor_p,
                                                  const int32_t *__restrict__ split_skip,
                                                  const int32_t *__restrict__ kept_rows,
                                                  const int64_t *__restrict__ kept_count,
                                                  int *__restrict__ queue) {
    using S = HopShape<BP>;
    const int lane = threadIdx.x & 31;
    const int sub = lane % S::LW;
    // with the skip (last hop), the rows kept whole that reach the floor
    // come as a compact list; a claim takes ROWS_PER_GRAB rows either way
    const bool listed = FILTER && kept_rows != nullptr;
    const int64_t grab = ROWS_PER_GRAB;
    const int64_t n_items = listed ? *kept_count : n;
    const int64_t groups = (n_items + grab - 1) / grab;
    __shared__ unsigned long long thr[FILTER ? BP : 1];
    __shared__ uint4 thr_hi[FILTER ? BP / 4 : 1];
    // last hop: rows whose bound stays below the floor append nothing
    const bool prune = FILTER && row_ub != nullptr;
    if constexpr (FILTER) {
        for (int c = threadIdx.x; c < BP; c += blockDim.x) {
            const unsigned long long t = f.bound[c];
            thr[c] = t;
            reinterpret_cast<uint32_t *>(thr_hi)[c] = (uint32_t)(t >> 32);
        }
        __syncthreads();
    }
    while (true) {
        int64_t it = 0;
        if (lane == 0) it = atomicAdd(queue, 1);
        it = __shfl_sync(0xffffffffu, it, 0);
        if (it >= n_split + groups) break;
        if (it < n_split) {
            const int32_t r = split_order[it];
            if (prune && split_skip[r]) continue;
            hop_fixup_row<BP, FILTER, WIDTH>(split_row[r], split_slot0[r], split_slot0[r + 1], part4,
                                      u4, out4, alpha, f, thr, thr_hi);
            continue;
        }
        // lane r: the claim's r-th row (consecutive rows, or listed ones),
        // its edge range; `todo`: the rows kept whole
        const int64_t i0 = (it - n_split) * grab;
        const int nr = (int)(n_items - i0 < grab ? n_items - i0 : grab);
        int64_t myrow = 0, p0 = 0, p1 = 0;
        if (lane < nr) {
            myrow = listed ? (int64_t)kept_rows[i0 + lane] : i0 + lane;
            p0 = in_ptr[myrow];
            p1 = in_ptr[myrow + 1];
        }
        const bool want = lane < nr && p1 - p0 <= split_t;
        unsigned todo = __ballot_sync(0xffffffffu, want);
        int32_t ids = 0;
        if (FILTER && want) ids = f.ext_of[myrow];
#pragma unroll 1
        while (todo) {
            const int r = __ffs(todo) - 1;
            todo &= todo - 1;
            const int64_t e0 = __shfl_sync(0xffffffffu, p0, r);
            const int64_t e1 = __shfl_sync(0xffffffffu, p1, r);
            const uint32_t id = FILTER ? (uint32_t)__shfl_sync(0xffffffffu, ids, r) : 0u;
            const int64_t j = __shfl_sync(0xffffffffu, myrow, r);
            float4 b[S::V];
            if (lane < S::LW) {
#pragma unroll
                for (int v = 0; v < S::V; ++v) b[v] = ld_stream(u4 + j * S::F + sub + 32 * v);
            }
            float4 acc[S::V];
            hop_accumulate<BP, WIDTH>(in_src, in_w, e0, e1, in4, acc);
            if (lane < S::LW) {
#pragma unroll
                for (int v = 0; v < S::V; ++v) {
                    b[v].x = fmaf(alpha, acc[v].x, b[v].x);
                    b[v].y = fmaf(alpha, acc[v].y, b[v].y);
                    b[v].z = fmaf(alpha, acc[v].z, b[v].z);
                    b[v].w = fmaf(alpha, acc[v].w, b[v].w);
                    if constexpr (!FILTER) st_stream(out4 + j * S::F + sub + 32 * v, b[v]);
                }
                hop_emit<BP, FILTER>(f, thr, thr_hi, sub, j, id, b);
            }
        }
    }
}

// Segments of split rows, claimed one at a time in window-major order.
template <int BP, int WIDTH = 1>
__global__ __launch_bounds__(256, WIDTH > 1 ? 2 : 3) void k_hop_segs(const int64_t *__restrict__ seg_e0,
                                                  const int64_t *__restrict__ seg_e1,
                                                  const int32_t *__restrict__ seg_slot,
                                                  int64_t n_segs,
                                                  const int32_t *__restrict__ in_src,
                                                  const float *__restrict__ in_w,
                                                  const float4 *__restrict__ in4,
                                                  float4 *__restrict__ part4,
                                                  const int32_t *__restrict__ kept_segs,
                                                  const int64_t *__restrict__ kept_count,
                                                  int *__restrict__ queue) {
    using S = HopShape<BP>;
    const int lane = threadIdx.x & 31;
    const int sub = lane % S::LW;
    // last hop: only the listed segments (those of unpruned split rows)
    const int64_t total = kept_segs ? *kept_count : n_segs;
    while (true) {
        int64_t i = 0;
        if (lane == 0) i = atomicAdd(queue, 1);
        i = __shfl_sync(0xffffffffu, i, 0);
        if (i >= total) break;
        const int64_t s = kept_segs ? (int64_t)kept_segs[i] : i;
        float4 acc[S::V];
        hop_accumulate<BP, WIDTH>(in_src, in_w, seg_e0[s], seg_e1[s], in4, acc);
        const int64_t slot = seg_slot[s];
        if (lane < S::LW) {
#pragma unroll
            for (int v = 0; v < S::V; ++v) st_stream(part4 + slot * S::F + sub + 32 * v, acc[v]);
        }
    }
}

template <int BP>
static cudaError_t hop_bp(const HopPlan &p, const float *u, const float *in, float *out,
                          float alpha, float *partial, int *counters, const HopFilter *flt,
                          cudaStream_t st, int *launches, const HopBound *hbp) {
    const int sms = device_sm_count();
    // the last hop skips rows whose bound stays below the filter floor
    const bool prune = flt && hbp && hbp->row_ub && hbp->floor && hbp->kept_rows &&
                       hbp->kept_count &&
                       (p.n_split_rows == 0 ||
                        (hbp->split_skip && hbp->slot_skip && hbp->kept_segs));
    cudaError_t e = cudaMemsetAsync(counters, 0, 2 * sizeof(int), st);
    if (e != cudaSuccess) return e;
    if (p.n_segs > 0) {
        const int64_t want = ceil_div<int64_t>(p.n_segs, 8);
        const int cps = prune ? 2 : 3;
        const int g2 = (int)(want < (int64_t)sms * cps ? want : (int64_t)sms * cps);
        if (prune)
            k_hop_segs<BP, 2><<<g2, 256, 0, st>>>(p.seg_e0, p.seg_e1, p.seg_slot, p.n_segs,
                                                  p.in_src, p.in_w, (const float4 *)in,
                                                  (float4 *)partial, hbp->kept_segs,
                                                  hbp->kept_count + 1, counters + 1);
        else
            k_hop_segs<BP><<<g2, 256, 0, st>>>(p.seg_e0, p.seg_e1, p.seg_slot, p.n_segs, p.in_src,
                                               p.in_w, (const float4 *)in, (float4 *)partial,
                                               nullptr, nullptr, counters + 1);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        if (launches) *launches += 1;
    }
    // (pruned: split rows + the kept list, its length known on the device only)
    const int64_t items = prune ? p.n_split_rows + 4096
                                : ceil_div<int64_t>(p.n, ROWS_PER_GRAB) + p.n_split_rows;
    const int64_t want = ceil_div<int64_t>(items, 8);
    const int cpr = prune ? 2 : 3;
    const int grid = (int)(want < (int64_t)sms * cpr ? (want < 1 ? 1 : want) : (int64_t)sms * cpr);
    const HopFilter f = flt ? *flt : HopFilter{nullptr, nullptr, nullptr, nullptr, 0, NsScope{}};
    if (prune)
        k_hop_rows<BP, true, 2><<<grid, 256, 0, st>>>(p.in_ptr, p.in_src, p.in_w, p.n,
                                                      (const float4 *)u, (const float4 *)in,
                                                      (float4 *)out, alpha, p.split.split_t,
                                                      p.n_split_rows, p.split_order, p.split_row,
                                                      p.split_slot0, (const float4 *)partial, f,
                                                      hbp->row_ub, hbp->floor, hbp->split_skip,
                                                      hbp->kept_rows, hbp->kept_count, counters);
    else if (flt)
        k_hop_rows<BP, true><<<grid, 256, 0, st>>>(p.in_ptr, p.in_src, p.in_w, p.n,
                                                   (const float4 *)u, (const float4 *)in,
                                                   (float4 *)out, alpha, p.split.split_t,
                                                   p.n_split_rows, p.split_order, p.split_row,
                                                   p.split_slot0, (const float4 *)partial, f,
                                                   nullptr, nullptr, nullptr, nullptr, nullptr,
                                                   counters);
    else
        k_hop_rows<BP, false><<<grid, 256, 0, st>>>(p.in_ptr, p.in_src, p.in_w, p.n,
                                                    (const float4 *)u, (const float4 *)in,
                                                    (float4 *)out, alpha, p.split.split_t,
                                                    p.n_split_rows, p.split_order, p.split_row,
                                                    p.split_slot0, (const float4 *)partial, f,
                                                    nullptr, nullptr, nullptr, nullptr, nullptr,
                                                    counters);
    if (launches) *launches += 1;
    return cudaGetLastError();
}

cudaError_t launch_hop(const HopPlan &p, const float *u, const float *in, float *out, int bp,
                       float alpha, float *partial, int *counters, const HopFilter *flt,
                       cudaStream_t st, int *launches, const HopBound *hb) {
    switch (bp) {
    case 32: return hop_bp<32>(p, u, in, out, alpha, partial, counters, flt, st, launches, hb);
    case 64: return hop_bp<64>(p, u, in, out, alpha, partial, counters, flt, st, launches, hb);
    case 128: return hop_bp<128>(p, u, in, out, alpha, partial, counters, flt, st, launches, hb);
    case 256: return hop_bp<256>(p, u, in, out, alpha, partial, counters, flt, st, launches, hb);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace ak
