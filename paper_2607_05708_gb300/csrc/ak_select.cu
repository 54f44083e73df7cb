// Top-k selection (a3) with score normalisation by Z (a1) and the page
// resolve + distinct-page count (a4): the top-p selection and FetchByID of
// query-aware retrieval (arXiv 2607.05708, §4.1, Algorithm 1) and the
// locality gap |P(R_t)| (§3.2).  The same machinery, on signed keys, selects
// the top-M prior chunks of the relation update.
//
// Three passes per batch of queries (columns of the score slab):
//   bound   the k-th largest value of every column over a strided sample
//           of the rows (a radix select per column).  A subset's k-th
//           largest value never exceeds the whole column's, so it is a safe
//           filter;
//   filter  one streaming pass over the slab (warp per row, coalesced
//           float4 loads) appending every key >= bound to a per-column
//           buffer;
//   merge   per column, an exact radix select of the k best buffered keys,
//           or of the whole column if the buffer overflowed.
#include "ak_common.cuh"

namespace ak {

constexpr int SEL_THREADS = 256;
constexpr int SEL_STAGE = 4096;   // keys a merge CTA stages in shared memory

// SIGNED=false: non-negative scores (retrieval); SIGNED=true: any finite
// value (cosines of the relation update).  Either way a larger key is a
// better candidate and equal values prefer the lower chunk ID.
template <bool SIGNED>
__device__ __forceinline__ unsigned long long sel_key(float v, uint32_t id) {
    const uint32_t hi = SIGNED ? ordered_bits(v) : __float_as_uint(v);
    return ((unsigned long long)hi << 32) | (unsigned long long)(~id);
}
template <bool SIGNED>
__device__ __forceinline__ float sel_value(unsigned long long key) {
    const uint32_t hi = (uint32_t)(key >> 32);
    return SIGNED ? unordered_bits(hi) : __uint_as_float(hi);
}

// ------------------------------------------------------------------ plan
SelectPlan select_plan(int64_t n, int bp, int k, int sm_count, int64_t force_stride) {
    SelectPlan sp;
    sp.n = n;
    sp.bp = bp;
    sp.k = k;
    // sample every stride-th row, at least 64 k rows (all rows of a small store)
    int64_t stride = n / ((int64_t)64 * k);
    stride = stride < 1 ? 1 : (stride > 32 ? 32 : stride);
    if (force_stride > 0) stride = force_stride;
    sp.stride = stride;
    sp.n_sample = ceil_div<int64_t>(n, stride);
    (void)sm_count;
    int64_t cap = 4 * (int64_t)k * stride;
    sp.cap = cap < 8192 ? 8192 : cap;
    sp.off_bound = 0;
    sp.off_cnt = sp.off_bound + bp;
    sp.off_buf = sp.off_cnt + bp;
    sp.off_tr = sp.off_buf + (int64_t)bp * sp.cap;
    sp.words = sp.off_tr + ceil_div<int64_t>(sp.n_sample * bp, 2);
    return sp;
}

// ------------------------------------------------------------------ radix select
// Exact k-th largest of `total` keys given by key_at(i), MSB-first 8 bits a
// pass with per-warp histograms; the (at most 64) keys >= it are left in
// win[] (unordered) and their count in *win_n.  Keys are unique apart from
// the padding key 0, which is below every real key and never selected.
template <typename KeyAt>
__device__ void radix_select(int64_t total, int k, KeyAt key_at, unsigned long long *win,
                             int *win_n, int *hist, unsigned long long *s_prefix,
                             int *s_remaining) {
    const int tid = threadIdx.x, warp = tid >> 5;
    if (tid == 0) {
        *s_prefix = 0ull;
        *s_remaining = k;
        *win_n = 0;
    }
    __syncthreads();
    unsigned long long pmask = 0ull;
    for (int pass = 0; pass < 8; ++pass) {
        const int sh = 56 - 8 * pass;
        for (int w = 0; w < SEL_THREADS / 32; ++w) hist[w * 256 + tid] = 0;
        __syncthreads();
        const unsigned long long prefix = *s_prefix;
        const int rem = *s_remaining;   // read before any thread can update it below
        for (int64_t i = tid; i < total; i += SEL_THREADS) {
            const unsigned long long key = key_at(i);
            if ((key & pmask) == prefix) atomicAdd(&hist[warp * 256 + ((key >> sh) & 0xff)], 1);
        }
        __syncthreads();
        // digit 255 - tid: its count and the inclusive count of all larger
        // digits (block-wide prefix sum), then the one thread whose range
        // holds the remaining rank records the digit
        int cntd = 0;
        for (int w = 0; w < SEL_THREADS / 32; ++w) cntd += hist[w * 256 + (255 - tid)];
        int incl = cntd;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, incl, o);
            if ((tid & 31) >= o) incl += t;
        }
        __syncthreads();
        if ((tid & 31) == 31) hist[tid >> 5] = incl;   // warp totals (hist is free now)
        __syncthreads();
        int before = 0;
        for (int w = 0; w < (tid >> 5); ++w) before += hist[w];
        incl += before;
        if (incl >= rem && incl - cntd < rem) {
            *s_remaining = rem - (incl - cntd);
            *s_prefix = prefix | ((unsigned long long)(255 - tid) << sh);
        }
        pmask |= 0xffull << sh;
        __syncthreads();
    }
    const unsigned long long kth = *s_prefix;
    for (int64_t i = tid; i < total; i += SEL_THREADS) {
        const unsigned long long key = key_at(i);
        if (key >= kth && key != 0ull) {
            const int p = atomicAdd(win_n, 1);
            if (p < 64) win[p] = key;
        }
    }
    __syncthreads();
}

// ------------------------------------------------------------------ bound pass
// bound[c] = the k-th largest sampled value of column c, as a key with the
// chunk-ID half zero (every key of that value clears it); 0 (admit all) if
// the sample holds fewer than k real values.  Sample rows are j = v*stride,
// v < n_sample; rows whose chunk ID is >= id_limit count as value-key 0.
constexpr int KTH_STAGE = 40960;   // sampled keys staged per CTA (160 KiB dynamic + ~49 KiB static)

// keysT[c][v] = key of sample row v in column c: 32 x 32 tiles through
// shared memory, so both the row reads and the column writes are
// coalesced.  Threads (tx, ty) = (tid % 32, tid / 32).
template <bool SIGNED>
__global__ __launch_bounds__(256) void k_sample_transpose(
    const float *__restrict__ s, int64_t n_sample, int64_t stride, int bp,
    const int32_t *__restrict__ ext_of, int64_t id_limit, NsScope ns,
    uint32_t *__restrict__ keysT) {
    __shared__ uint32_t tile[32][33];
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int64_t v0 = (int64_t)blockIdx.x * 32;
    const int c0 = blockIdx.y * 32;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int r = ty + 8 * i;
        const int64_t v = v0 + r;
        uint32_t key = 0u;
        if (v < n_sample) {
            const int64_t j = v * stride;
            if ((int64_t)ext_of[j] < id_limit && in_scope(ns, j, c0 + tx)) {
                const float x = s[j * bp + c0 + tx];
                key = SIGNED ? ordered_bits(x) : __float_as_uint(x);
            }
        }
        tile[r][tx] = key;
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int cc = ty + 8 * i;
        const int64_t v = v0 + tx;
        if (v < n_sample) keysT[(int64_t)(c0 + cc) * n_sample + v] = tile[tx][cc];
    }
}

// bound[c] from column c of keysT: staged in shared memory when it fits,
// then an MSB-first radix select over the bits below the column's common
// prefix (the sampled values of one column mostly share sign, exponent and
// leading mantissa bits, so starting below them both saves passes and
// spreads the first digit).  Histograms are replicated per warp and per
// lane quarter to cut shared-memory atomic contention on popular digits;
// every thread does the same work per key (no data-dependent loops).
constexpr int KTH_REP = (SEL_THREADS / 32) * 4;   // histogram replicas
constexpr int KTH_CBUF = 4096;                    // keys kept after the first digit

__global__ __launch_bounds__(SEL_THREADS) void k_sample_kth(
    const uint32_t *__restrict__ keysT, int64_t n_sample, int b, int k, uint32_t slack,
    unsigned long long *__restrict__ bound, unsigned int *__restrict__ cnt) {
    extern __shared__ uint32_t kst[];                 // [n_sample] when staged
    __shared__ int hist[KTH_REP * 256];
    __shared__ int wsum[SEL_THREADS / 32];
    __shared__ uint32_t red_or[SEL_THREADS / 32], red_and[SEL_THREADS / 32];
    __shared__ uint32_t cbuf[KTH_CBUF];
    __shared__ uint32_t s_prefix;
    __shared__ int s_rem, s_match, s_cn;
    const int c = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (c >= b) {   // padding column: nothing passes the filter
        if (tid == 0) {
            bound[c] = ~0ull;
            cnt[c] = 0u;
        }
        return;
    }
    const uint32_t *col = keysT + (int64_t)c * n_sample;
    const bool staged = n_sample <= KTH_STAGE;
    // stage, and find the bits on which the column's keys differ
    uint32_t k_or = 0u, k_and = ~0u;
    for (int64_t v = tid; v < n_sample; v += SEL_THREADS) {
        const uint32_t x = col[v];
        if (staged) kst[v] = x;
        k_or |= x;
        k_and &= x;
    }
    for (int o = 16; o > 0; o >>= 1) {
        k_or |= __shfl_xor_sync(0xffffffffu, k_or, o);
        k_and &= __shfl_xor_sync(0xffffffffu, k_and, o);
    }
    if (lane == 0) {
        red_or[warp] = k_or;
        red_and[warp] = k_and;
    }
    __syncthreads();
    k_or = 0u;
    k_and = ~0u;
    for (int w = 0; w < SEL_THREADS / 32; ++w) {
        k_or |= red_or[w];
        k_and &= red_and[w];
    }
    const uint32_t diff = k_or & ~k_and;              // bits that vary
    const int top0 = diff ? 31 - __clz(diff) : -1;    // highest varying bit
    // bits above top0, identical in every key (all bits if no bit varies)
    const uint32_t above = top0 < 0 ? ~0u : (top0 == 31 ? 0u : ~((2u << top0) - 1u));
    const uint32_t common = k_and & above;
    if (tid == 0) {
        s_prefix = common;
        s_rem = k;
    }
    __syncthreads();
    uint32_t pmask = above;                           // bits fixed so far
    const int hrep = (warp * 4 + (lane & 3)) * 256;
    // keys still in play: the whole column, and after a digit that leaves
    // at most KTH_CBUF candidates, just those (compacted into cbuf)
    const uint32_t *keys = staged ? kst : col;
    int64_t len = n_sample;
    for (int top = top0; top >= 0; top -= 8) {
        const int sh = top >= 7 ? top - 7 : 0;
        const uint32_t dmask = (2u << (top - sh)) - 1u;
        for (int i = tid; i < KTH_REP * 256; i += SEL_THREADS) hist[i] = 0;
        __syncthreads();
        const uint32_t prefix = s_prefix;
        const int rem = s_rem;
        for (int64_t v = tid; v < len; v += SEL_THREADS) {
            const uint32_t key = keys[v];
            if ((key & pmask) == prefix) atomicAdd(&hist[hrep + ((key >> sh) & dmask)], 1);
        }
        __syncthreads();
        // thread t owns digit 255 - t: its count and the inclusive count of
        // all larger digits; the thread whose range holds rank `rem` wins
        int cntd = 0;
        for (int r = 0; r < KTH_REP; ++r) cntd += hist[r * 256 + (255 - tid)];
        int incl = cntd;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += t;
        }
        if (lane == 31) wsum[warp] = incl;
        __syncthreads();
        for (int w = 0; w < warp; ++w) incl += wsum[w];
        if (incl >= rem && incl - cntd < rem) {
            s_rem = rem - (incl - cntd);
            s_prefix = prefix | ((uint32_t)(255 - tid) << sh);
            s_match = cntd;
        }
        pmask |= dmask << sh;
        if (tid == 0) s_cn = 0;
        __syncthreads();
        if (sh > 0 && len > KTH_CBUF && n_sample >= k && s_match <= KTH_CBUF) {
            const uint32_t pre = s_prefix;
            for (int64_t v = tid; v < len; v += SEL_THREADS) {
                const uint32_t key = keys[v];
                if ((key & pmask) == pre) cbuf[atomicAdd(&s_cn, 1)] = key;
            }
            __syncthreads();
            keys = cbuf;
            len = s_match;
        }
    }
    if (tid == 0) {
        // fewer than k keys: no thread ever matched and the prefix has not
        // reached a key, so admit everything
        const bool found = n_sample >= k;
        const uint32_t kth = s_prefix > slack ? s_prefix - slack : 0u;
        bound[c] = found ? (unsigned long long)kth << 32 : 0ull;
        cnt[c] = 0u;
    }
}

// bound[c] from column c of keys_t, split over KS_WARPS warps.  Each warp
// scans a contiguous share of the column and keeps, in its own shared
// buffer, every key above a running threshold t (0 at first: key 0 marks a
// row that is out of the selection).  When the buffer is full it is cut to
// its k largest keys (the keys above its k-th largest key x, then copies of
// x up to k) and t becomes x: every key outside the buffer is then <= t <=
// every key inside, so the k-th largest of the buffer stays the k-th
// largest of the warp's share.  At the end each warp cuts its buffer to at
// most k keys, and warp 0 selects the k-th largest of their union.
constexpr int KS_WARPS = 4, KS_BUF = 512, KS_U = 16, KS_KMAX = 64;

// The k-th largest (1 <= k <= len <= KS_BUF) of a[0..len) by one warp: the
// keys in registers (KS_BUF / 32 a lane, 0 past len, which ranks below
// every candidate), then the answer's bits from the top, each kept when at
// least k keys are >= the prefix with it set (the largest t with k keys
// >= t is the k-th largest key).  No shared-memory atomics: the sampled
// keys of one column share their top bits, so histogram bins would collide.
__device__ __noinline__ uint32_t warp_kth(const uint32_t *a, int len, int k) {
    const int lane = threadIdx.x & 31;
    uint32_t x[KS_BUF / 32];
#pragma unroll
    for (int j = 0; j < KS_BUF / 32; ++j) {
        const int i = j * 32 + lane;
        x[j] = i < len ? a[i] : 0u;
    }
    uint32_t prefix = 0u;
#pragma unroll 1
    for (int b = 31; b >= 0; --b) {
        const uint32_t cand = prefix | (1u << b);
        unsigned c = 0u;
#pragma unroll
        for (int j = 0; j < KS_BUF / 32; ++j) c += x[j] >= cand ? 1u : 0u;
        c = __reduce_add_sync(0xffffffffu, c);
        if (c >= (unsigned)k) prefix = cand;
    }
    return prefix;
}

// Cut a[0..len) (len >= k) to its k largest; returns the k-th largest.
// (Called out of line from the scan's unrolled loop, which it would
// otherwise bloat past the instruction cache.)
__device__ __noinline__ uint32_t warp_cut(uint32_t *a, int len, int k) {
    const int lane = threadIdx.x & 31;
    const unsigned lt = (1u << lane) - 1u;
    const uint32_t x = warp_kth(a, len, k);
    int out = 0;
    for (int i0 = 0; i0 < len; i0 += 32) {
        const uint32_t v = i0 + lane < len ? a[i0 + lane] : 0u;
        const bool keep = i0 + lane < len && v > x;
        const unsigned bal = __ballot_sync(0xffffffffu, keep);
        __syncwarp();
        if (keep) a[out + __popc(bal & lt)] = v;   // out + rank <= i0 + lane: already read
        out += __popc(bal);
        __syncwarp();
    }
    for (int j = out + lane; j < k; j += 32) a[j] = x;
    __syncwarp();
    return x;
}

__global__ __launch_bounds__(KS_WARPS * 32) void k_sample_kth_split(
    const uint32_t *__restrict__ keys_t, int64_t n_sample, int b, int k,
    unsigned long long *__restrict__ bound, unsigned int *__restrict__ cnt) {
    __shared__ uint32_t buf[KS_WARPS][KS_BUF];
    __shared__ int lens[KS_WARPS];
    const int c = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (c >= b) {   // padding column: nothing passes the filter
        if (threadIdx.x == 0) {
            bound[c] = ~0ull;
            cnt[c] = 0u;
        }
        return;
    }
    const unsigned lt = (1u << lane) - 1u;
    const uint32_t *col = keys_t + (int64_t)c * n_sample;
    const int64_t share = (n_sample + KS_WARPS - 1) / KS_WARPS;
    const int64_t v_lo = warp * share;
    const int64_t v_hi = v_lo + share < n_sample ? v_lo + share : n_sample;
    uint32_t *a = buf[warp];
    uint32_t t = 0u;
    int len = 0;
    for (int64_t v0 = v_lo; v0 < v_hi; v0 += 32 * KS_U) {
        uint32_t x[KS_U];
#pragma unroll
        for (int u = 0; u < KS_U; ++u) {
            const int64_t v = v0 + u * 32 + lane;
            x[u] = v < v_hi ? __ldcs(col + v) : 0u;
        }
#pragma unroll
        for (int u = 0; u < KS_U; ++u) {
            const bool p = x[u] > t;
            const unsigned bal = __ballot_sync(0xffffffffu, p);
            if (bal) {
                if (len + 32 > KS_BUF) {
                    t = warp_cut(a, len, k);
                    len = k;
                }
                const bool q = p && x[u] > t;       // the cut may have raised t
                const unsigned bq = __ballot_sync(0xffffffffu, q);
                if (q) a[len + __popc(bq & lt)] = x[u];
                len += __popc(bq);
                __syncwarp();
            }
        }
    }
    if (len > k) {
        warp_cut(a, len, k);
        len = k;
    }
    if (lane == 0) lens[warp] = len;
    __syncthreads();
    if (warp == 0) {
        // the survivors of all warps, gathered behind warp 0's own
        int tot = lens[0];
        for (int w = 1; w < KS_WARPS; ++w) {
            for (int i = lane; i < lens[w]; i += 32) a[tot + i] = buf[w][i];
            tot += lens[w];
        }
        __syncwarp();
        const uint32_t x = tot >= k ? warp_kth(a, tot, k) : 0u;
        if (lane == 0) {
            bound[c] = (unsigned long long)x << 32;
            cnt[c] = 0u;
        }
    }
}

cudaError_t launch_sample_kth_keys(const uint32_t *keys_t, int64_t n_sample, int bp, int b, int k,
                                   unsigned long long *bound, unsigned int *cnt, cudaStream_t st,
                                   int *launches) {
    if (k < 1 || k > KS_KMAX || bp < 1 || b > bp || KS_WARPS * KS_KMAX > KS_BUF)
        return cudaErrorInvalidValue;
    k_sample_kth_split<<<bp, KS_WARPS * 32, 0, st>>>(keys_t, n_sample, b, k, bound, cnt);
    if (launches) *launches += 1;
    return cudaGetLastError();
}

// ------------------------------------------------------------------ filter pass
template <int BP>
struct SelShape {
    static constexpr int F = BP / 4;                 // float4 per row
    static constexpr int G = F >= 32 ? 1 : 32 / F;   // rows per warp step
    static constexpr int V = F >= 32 ? F / 32 : 1;   // float4 per lane
    static constexpr int LW = F >= 32 ? 32 : F;      // lanes per row
};

// Append key to column c's buffer if it clears the bound.
__device__ __forceinline__ void sel_push(unsigned long long key, unsigned long long bound, int c,
                                         unsigned int *__restrict__ cnt,
                                         unsigned long long *__restrict__ buf, int64_t cap,
                                         const NsScope &ns, int64_t j) {
    if (key >= bound && in_scope(ns, j, c)) {
        const unsigned int p = atomicAdd(&cnt[c], 1u);
        if ((int64_t)p < cap) buf[(int64_t)c * cap + p] = key;
    }
}

template <int BP, bool SIGNED>
__global__ __launch_bounds__(256) void k_filter(const float *__restrict__ s, int64_t n,
                                                const int32_t *__restrict__ ext_of,
                                                int64_t id_limit, NsScope ns,
                                                const unsigned long long *__restrict__ bound,
                                                unsigned int *__restrict__ cnt,
                                                unsigned long long *__restrict__ buf, int64_t cap) {
    using S = SelShape<BP>;
    constexpr int R = 4;   // row steps in flight per warp
    const int lane = threadIdx.x & 31;
    const int g = lane / S::LW, sub = lane % S::LW;
    unsigned long long thr[S::V][4];
#pragma unroll
    for (int v = 0; v < S::V; ++v)
#pragma unroll
        for (int e = 0; e < 4; ++e) thr[v][e] = bound[(sub + 32 * v) * 4 + e];
    const float4 *s4 = (const float4 *)s;
    const int64_t steps = (n + S::G - 1) / S::G;
    const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t t0 = warp * R; t0 < steps; t0 += nwarps * R) {
        float4 x[R][S::V];
        int32_t id[R];
#pragma unroll
        for (int q = 0; q < R; ++q) {
            const int64_t j = (t0 + q) * S::G + g;
            const bool ok = t0 + q < steps && j < n;
            id[q] = ok ? ext_of[j] : (int32_t)0x7fffffff;
#pragma unroll
            for (int v = 0; v < S::V; ++v)
                x[q][v] = ok ? s4[j * S::F + sub + 32 * v] : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int q = 0; q < R; ++q) {
            if ((int64_t)id[q] >= id_limit) continue;
            const uint32_t u = (uint32_t)id[q];
            const int64_t j = (t0 + q) * S::G + g;
#pragma unroll
            for (int v = 0; v < S::V; ++v) {
                const int c = (sub + 32 * v) * 4;
                sel_push(sel_key<SIGNED>(x[q][v].x, u), thr[v][0], c, cnt, buf, cap, ns, j);
                sel_push(sel_key<SIGNED>(x[q][v].y, u), thr[v][1], c + 1, cnt, buf, cap, ns, j);
                sel_push(sel_key<SIGNED>(x[q][v].z, u), thr[v][2], c + 2, cnt, buf, cap, ns, j);
                sel_push(sel_key<SIGNED>(x[q][v].w, u), thr[v][3], c + 3, cnt, buf, cap, ns, j);
            }
        }
    }
}

// ------------------------------------------------------------------ merge pass
// The k best keys of column c: from its buffer (staged in shared memory when
// small), or from the whole column of the slab if the buffer overflowed.
template <bool SIGNED>
__device__ void column_top(const float *__restrict__ s, int64_t n, int bp, int k, int c,
                           const int32_t *__restrict__ ext_of, int64_t id_limit,
                           const unsigned int *__restrict__ cnt,
                           const unsigned long long *__restrict__ buf, int64_t cap,
                           unsigned long long *stage, unsigned long long *win, int *win_n,
                           int *hist, unsigned long long *s_prefix, int *s_remaining,
                           NsScope ns = NsScope{}) {
    const int64_t m = cnt[c];
    if (m <= SEL_THREADS) {
        // few candidates: each thread ranks one key against the others (the
        // keys are unique but for the padding 0, never selected), and the
        // keys ranked below k are the ones radix_select would leave in win[]
        const unsigned long long *bc = buf + (int64_t)c * cap;
        const int tid = threadIdx.x;
        if (tid == 0) *win_n = 0;
        if (tid < m) stage[tid] = bc[tid];
        __syncthreads();
        if (tid < m) {
            const unsigned long long x = stage[tid];
            if (x != 0ull) {
                int r = 0;
                for (int j = 0; j < (int)m; ++j) r += stage[j] > x ? 1 : 0;
                if (r < k) {
                    const int p = atomicAdd(win_n, 1);
                    if (p < 64) win[p] = x;
                }
            }
        }
        __syncthreads();
        return;
    }
    if (m <= cap) {
        const unsigned long long *bc = buf + (int64_t)c * cap;
        if (m <= SEL_STAGE) {
            for (int64_t i = threadIdx.x; i < m; i += SEL_THREADS) stage[i] = bc[i];
            __syncthreads();
            auto key_at = [&](int64_t i) -> unsigned long long { return stage[i]; };
            radix_select(m, k, key_at, win, win_n, hist, s_prefix, s_remaining);
        } else {
            auto key_at = [&](int64_t i) -> unsigned long long { return bc[i]; };
            radix_select(m, k, key_at, win, win_n, hist, s_prefix, s_remaining);
        }
    } else {
        auto key_at = [&](int64_t i) -> unsigned long long {
            const int32_t id = ext_of[i];
            return ((int64_t)id >= id_limit || !in_scope(ns, i, c))
                       ? 0ull : sel_key<SIGNED>(s[i * bp + c], (uint32_t)id);
        };
        radix_select(n, k, key_at, win, win_n, hist, s_prefix, s_remaining);
    }
}

// Retrieval merge, one CTA per real query column: the k winners ordered by
// key (score desc, id asc), normalised by Z = sum of the score pass's
// partials, resolved to pages, and their distinct pages counted.
__global__ __launch_bounds__(SEL_THREADS) void k_topk_merge(
    const float *__restrict__ s, int64_t n, int bp, int k, const int32_t *__restrict__ ext_of,
    const unsigned int *__restrict__ cnt, const unsigned long long *__restrict__ buf, int64_t cap,
    const float *__restrict__ zpart, int64_t n_ztiles, const int32_t *__restrict__ row_of,
    const int32_t *__restrict__ page_row, int64_t *__restrict__ ids, float *__restrict__ scores,
    int32_t *__restrict__ page_ids, int32_t *__restrict__ n_pages, int *status,
    const ColumnRecompute rc, const NsScope ns, const int sort_by_time) {
    __shared__ int hist[256 * (SEL_THREADS / 32)];
    __shared__ unsigned long long stage[SEL_STAGE];
    __shared__ unsigned long long win[64];
    __shared__ unsigned long long s_prefix;
    __shared__ int s_remaining, win_n;
    __shared__ double zred[SEL_THREADS / 32];
    __shared__ int pg[64];
    griddep_wait();
    const int c = blockIdx.x;
    const int tid = threadIdx.x;
    if (rc.kind != 0 && (int64_t)cnt[c] > cap) {
        // the buffer overflowed and no slab holds the final column:
        // recompute it (warp per row; lanes over the row's in-edges for the
        // last hop, over the embedding for the score)
        const int lane = tid & 31;
        for (int64_t j = tid >> 5; j < n; j += SEL_THREADS / 32) {
            float acc = 0.f;
            if (rc.kind == 1) {
                for (int64_t e = rc.in_ptr[j] + lane; e < rc.in_ptr[j + 1]; e += 32)
                    acc = fmaf(rc.in_w[e], rc.prev[(int64_t)rc.in_src[e] * bp + c], acc);
            } else {
                const uint16_t *ej = rc.emb + j * rc.dim, *qc = rc.qp + (int64_t)c * rc.dim;
                for (int t = lane; t < rc.dim; t += 32)
                    acc = fmaf(bf16_to_f32(ej[t]), bf16_to_f32(qc[t]), acc);
            }
            for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
            if (lane == 0)
                rc.dst[j * bp + c] = rc.kind == 1 ? fmaf(rc.alpha, acc, rc.u[j * bp + c])
                                                  : exp2f(fmaf(acc, rc.tau * LOG2E_F,
                                                               -rc.shift[c] * LOG2E_F));
        }
        __threadfence_block();
        __syncthreads();
    }
    double z = 0.0;
    for (int64_t t = tid; t < n_ztiles; t += SEL_THREADS) z += (double)zpart[t * bp + c];
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    if ((tid & 31) == 0) zred[tid >> 5] = z;
    column_top<false>(s, n, bp, k, c, ext_of, (int64_t)1 << 40, cnt, buf, cap, stage, win, &win_n,
                      hist, &s_prefix, &s_remaining, ns);
    // without a scope every query has k winners; with one, a namespace
    // holding fewer than k chunks pads its list
    if (tid == 0 && (win_n > k || (!scope_active(ns) && win_n != k)))
        set_status(status, AKASHIC_EDEVICE);
    const int got = win_n < k ? win_n : k;
    if (tid < got) {
        const unsigned long long key = win[tid];
        const uint32_t id = key_id(key);
        // rank by score (key desc) or, with SortByTime, by chunk ID
        int rank = 0;
        for (int t = 0; t < got; ++t)
            rank += sort_by_time ? (key_id(win[t]) < id) : (win[t] > key);
        double zsum = 0.0;
        for (int w = 0; w < SEL_THREADS / 32; ++w) zsum += zred[w];
        const int64_t o = (int64_t)c * k + rank;
        ids[o] = (int64_t)id;
        scores[o] = (float)((double)sel_value<false>(key) / zsum);
        const int32_t p = page_row ? page_row[row_of[id]] : 0;
        pg[rank] = p;
        if (page_ids) page_ids[o] = p;
    } else if (tid < k) {
        const int64_t o = (int64_t)c * k + tid;
        ids[o] = -1;
        scores[o] = 0.f;
        if (page_ids) page_ids[o] = -1;
    }
    __syncthreads();
    if (n_pages && tid < 32) {
        int distinct = 0;
        for (int a = tid; a < got; a += 32) {
            bool first = true;
            for (int b2 = 0; b2 < a; ++b2) first &= pg[b2] != pg[a];
            distinct += first;
        }
        for (int o = 16; o > 0; o >>= 1) distinct += __shfl_xor_sync(0xffffffffu, distinct, o);
        if (tid == 0) n_pages[c] = distinct;
    }
}

// Relation-update merge: the M best prior chunks of new chunk c (ordered by
// cosine desc, id asc) into nbr_ids / nbr_cos rows c_base + c.
__global__ __launch_bounds__(SEL_THREADS) void k_topm_merge(
    const float *__restrict__ s, int64_t n, int bp, int k, const int32_t *__restrict__ ext_of,
    int64_t id_limit, const unsigned int *__restrict__ cnt,
    const unsigned long long *__restrict__ buf, int64_t cap, int64_t c_base,
    int32_t *__restrict__ nbr_ids, float *__restrict__ nbr_cos, int *status, const NsScope ns) {
    __shared__ int hist[256 * (SEL_THREADS / 32)];
    __shared__ unsigned long long stage[SEL_STAGE];
    __shared__ unsigned long long win[64];
    __shared__ unsigned long long s_prefix;
    __shared__ int s_remaining, win_n;
    const int c = blockIdx.x;
    const int tid = threadIdx.x;
    column_top<true>(s, n, bp, k, c, ext_of, id_limit, cnt, buf, cap, stage, win, &win_n, hist,
                     &s_prefix, &s_remaining, ns);
    if (tid == 0 && win_n != k) set_status(status, AKASHIC_EDEVICE);
    const int got = win_n < k ? win_n : k;
    if (tid < got) {
        const unsigned long long key = win[tid];
        int rank = 0;
        for (int t = 0; t < got; ++t) rank += win[t] > key;
        const int64_t o = (c_base + c) * k + rank;
        nbr_ids[o] = (int32_t)key_id(key);
        nbr_cos[o] = sel_value<true>(key);
    }
}

// Relation top-M from the fused filter's buffers alone (one CTA per new
// chunk c; the caller has checked that no buffer overflowed).
__global__ __launch_bounds__(SEL_THREADS) void k_buf_merge_signed(
    const unsigned int *__restrict__ cnt, const unsigned long long *__restrict__ buf, int64_t cap,
    int k, int32_t *__restrict__ nbr_ids, float *__restrict__ nbr_cos, int *status) {
    __shared__ int hist[256 * (SEL_THREADS / 32)];
    __shared__ unsigned long long stage[SEL_STAGE];
    __shared__ unsigned long long win[64];
    __shared__ unsigned long long s_prefix;
    __shared__ int s_remaining, win_n;
    const int64_t c = blockIdx.x;
    const int tid = threadIdx.x;
    const int64_t m = cnt[c] < cap ? cnt[c] : cap;
    const unsigned long long *bc = buf + c * cap;
    if (m <= SEL_STAGE) {
        for (int64_t i = tid; i < m; i += SEL_THREADS) stage[i] = bc[i];
        __syncthreads();
        auto key_at = [&](int64_t i) -> unsigned long long { return stage[i]; };
        radix_select(m, k, key_at, win, &win_n, hist, &s_prefix, &s_remaining);
    } else {
        auto key_at = [&](int64_t i) -> unsigned long long { return bc[i]; };
        radix_select(m, k, key_at, win, &win_n, hist, &s_prefix, &s_remaining);
    }
    if (tid == 0 && win_n != k) set_status(status, AKASHIC_EDEVICE);
    const int got = win_n < k ? win_n : k;
    if (tid < got) {
        const unsigned long long key = win[tid];
        int rank = 0;
        for (int t = 0; t < got; ++t) rank += win[t] > key;
        nbr_ids[c * k + rank] = (int32_t)key_id(key);
        nbr_cos[c * k + rank] = sel_value<true>(key);
    }
}

cudaError_t launch_buf_merge_signed(const unsigned int *cnt, const unsigned long long *buf,
                                    int64_t cap, int64_t n_cols, int k, int32_t *nbr_ids,
                                    float *nbr_cos, int *status, cudaStream_t st, int *launches) {
    if (n_cols <= 0) return cudaSuccess;
    k_buf_merge_signed<<<(unsigned)n_cols, SEL_THREADS, 0, st>>>(cnt, buf, cap, k, nbr_ids,
                                                                 nbr_cos, status);
    if (launches) *launches += 1;
    return cudaGetLastError();
}

// ------------------------------------------------------------------ last-hop floor
// The smallest final score any real query could still select: the largest of
// (a) the smallest score bits that any real column's filter bound admits
// (keys of non-negative scores order like their values; padding bounds,
// above +inf's bits, admit nothing) and (b), without a namespace scope, the
// k-th largest lower bound lb over the rows lb_rows[order[i]], i < n_rows
// (at most PF_ROWS): every query's k-th largest final score is at least
// that, as each of those k rows scores at least its lb for every query (any
// subset of the rows gives a valid floor).  One CTA, one key per thread:
// (b) sorts the unique keys (lb bits, position) descending with a bitonic
// network (partners within a warp by shuffles, farther ones through a
// ping-pong pair of shared arrays) and reads the k-th.
constexpr int PF_ROWS = 1024;

__global__ __launch_bounds__(PF_ROWS) void k_prune_floor(
    const unsigned long long *__restrict__ bound, int n_real, const float *__restrict__ lb,
    const int32_t *__restrict__ lb_rows, const int32_t *__restrict__ order, int64_t n_rows,
    int k, float *__restrict__ floor_out) {
    __shared__ unsigned long long xk[2][PF_ROWS];
    __shared__ unsigned int s_min;
    const int t = threadIdx.x;
    if (t == 0) s_min = 0x7f800000u;
    __syncthreads();
    if (bound && t < n_real) atomicMin(&s_min, (unsigned int)(bound[t] >> 32));
    const bool want_lb = lb_rows && n_rows >= k;
    // absent keys are 0, below every real key but (lb = 0, position 0),
    // which they equal
    unsigned long long key =
        want_lb && t < n_rows
            ? ((unsigned long long)__float_as_uint(lb[lb_rows[order[t]]]) << 32) |
                  (unsigned long long)(uint32_t)t
            : 0ull;
    int cur = 0;
    if (want_lb) {
        for (int size = 2; size <= PF_ROWS; size <<= 1) {
            for (int stride = size >> 1; stride > 0; stride >>= 1) {
                unsigned long long other;
                if (stride >= 32) {
                    xk[cur][t] = key;
                    __syncthreads();
                    other = xk[cur][t ^ stride];
                    cur ^= 1;          // the next write goes to the other array
                } else {
                    other = __shfl_xor_sync(0xffffffffu, key, stride);
                }
                // segments with (t & size) == 0 run descending: there the
                // lower position of each pair keeps the larger key
                const bool keep_max = ((t & size) == 0) == ((t & stride) == 0);
                key = keep_max ? (key > other ? key : other) : (key < other ? key : other);
            }
        }
        if (t == k - 1) xk[cur][0] = key;
    }
    __syncthreads();
    if (t == 0) {
        // without filter bounds (no first term) the floor starts at 0
        float fl = bound ? __uint_as_float(s_min) : 0.f;
        if (want_lb) fl = fmaxf(fl, __uint_as_float((uint32_t)(xk[cur][0] >> 32)));
        *floor_out = fl;
    }
}

// The batch's distinct query namespaces, ascending, and for each the
// smallest score that the filter bound of any of its queries admits.  One
// CTA of PF_TAGS threads: keys (valid, tag) sorted by a bitonic network in
// shared memory, first occurrences numbered by a scan.
__global__ __launch_bounds__(PF_TAGS) void k_ns_tags(const unsigned long long *__restrict__ bound,
                                                     const int32_t *__restrict__ q_ns, int n_real,
                                                     int32_t *__restrict__ tags,
                                                     int *__restrict__ n_tags,
                                                     float *__restrict__ tag_floor) {
    __shared__ unsigned long long key[PF_TAGS];
    __shared__ int pos[PF_TAGS];
    __shared__ unsigned int mn[PF_TAGS];
    const int t = threadIdx.x;
    // valid tags first, in signed order; padding (1 << 32) last
    key[t] = t < n_real ? (unsigned long long)((uint32_t)q_ns[t] ^ 0x80000000u) : (1ull << 32);
    mn[t] = 0x7f800000u;
    __syncthreads();
    for (int size = 2; size <= PF_TAGS; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const int o = t ^ stride;
            if (o > t) {
                const unsigned long long a = key[t], b = key[o];
                const bool asc = (t & size) == 0;
                if (asc ? a > b : a < b) {
                    key[t] = b;
                    key[o] = a;
                }
            }
            __syncthreads();
        }
    const bool first = key[t] < (1ull << 32) && (t == 0 || key[t - 1] != key[t]);
    pos[t] = first ? 1 : 0;
    __syncthreads();
    for (int o = 1; o < PF_TAGS; o <<= 1) {          // inclusive scan
        const int v = t >= o ? pos[t - o] : 0;
        __syncthreads();
        pos[t] += v;
        __syncthreads();
    }
    const int nt = pos[PF_TAGS - 1];
    if (first) tags[pos[t] - 1] = (int32_t)((uint32_t)key[t] ^ 0x80000000u);
    if (t == 0) *n_tags = nt;
    __syncthreads();
    if (t < n_real && bound) {
        const int32_t mine = q_ns[t];
        int lo = 0, hi = nt;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (tags[mid] < mine) lo = mid + 1;
            else hi = mid;
        }
        atomicMin(&mn[lo], (unsigned int)(bound[t] >> 32));
    }
    __syncthreads();
    if (t < nt) tag_floor[t] = bound ? __uint_as_float(mn[t]) : 0.f;
}

// tag_floor[d] = max(tag_floor[d], k-th largest lb over the first PF_ROWS
// split rows, heaviest first, of namespace tags[d]); one CTA per tag.
__global__ __launch_bounds__(PF_ROWS) void k_ns_floor(const float *__restrict__ lb,
                                                      const int32_t *__restrict__ ns_row,
                                                      const int32_t *__restrict__ split_row,
                                                      const int32_t *__restrict__ order,
                                                      int64_t n_split, int k,
                                                      const int32_t *__restrict__ tags,
                                                      const int *__restrict__ n_tags,
                                                      float *__restrict__ tag_floor) {
    __shared__ unsigned int key[PF_ROWS];
    __shared__ int wcount[PF_ROWS / 32];
    __shared__ int got_s;
    const int d = blockIdx.x;
    if (d >= *n_tags) return;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    const int32_t tag = tags[d];
    key[t] = 0u;
    if (t == 0) got_s = 0;
    __syncthreads();
    for (int64_t c0 = 0; c0 < n_split; c0 += PF_ROWS) {
        const int got = got_s;
        if (got >= PF_ROWS) break;
        const int64_t i = c0 + t;
        int32_t r = 0;
        const bool match = i < n_split && ns_row[r = split_row[order[i]]] == tag;
        const unsigned int bal = __ballot_sync(0xffffffffu, match);
        if (lane == 0) wcount[w] = __popc(bal);
        __syncthreads();
        int before = got;
        for (int x = 0; x < w; ++x) before += wcount[x];
        before += __popc(bal & ((1u << lane) - 1u));
        if (match && before < PF_ROWS) key[before] = __float_as_uint(lb[r]);   // lb >= 0
        __syncthreads();
        if (t == 0) {
            int tot = got;
            for (int x = 0; x < PF_ROWS / 32; ++x) tot += wcount[x];
            got_s = tot;
        }
        __syncthreads();
    }
    const int got = got_s < PF_ROWS ? got_s : PF_ROWS;
    if (got < k) return;                              // too few rows for a floor of their own
    // descending bitonic sort of the collected keys (absent ones are 0)
    for (int size = 2; size <= PF_ROWS; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const int o = t ^ stride;
            if (o > t) {
                const unsigned int a = key[t], b = key[o];
                const bool desc = (t & size) == 0;
                if (desc ? a < b : a > b) {
                    key[t] = b;
                    key[o] = a;
                }
            }
            __syncthreads();
        }
    if (t == 0) tag_floor[d] = fmaxf(tag_floor[d], __uint_as_float(key[k - 1]));
}

cudaError_t launch_ns_floors(const unsigned long long *bound, const int32_t *q_ns, int n_real,
                             const float *lb, const int32_t *ns_row, const int32_t *split_row,
                             const int32_t *split_order, int64_t n_split, int k, int32_t *tags,
                             int *n_tags, float *tag_floor, cudaStream_t st) {
    if (n_real < 1 || n_real > PF_TAGS || k < 1) return cudaErrorInvalidValue;
    k_ns_tags<<<1, PF_TAGS, 0, st>>>(bound, q_ns, n_real, tags, n_tags, tag_floor);
    if (n_split > 0 && k <= PF_ROWS)
        k_ns_floor<<<PF_TAGS, PF_ROWS, 0, st>>>(lb, ns_row, split_row, split_order, n_split, k,
                                                tags, n_tags, tag_floor);
    return cudaGetLastError();
}

cudaError_t launch_prune_floor(const unsigned long long *bound, int n_real, const float *lb,
                               const int32_t *lb_rows, const int32_t *order, int64_t n_lb_rows,
                               int k, float *floor_out, cudaStream_t st) {
    if (n_lb_rows > PF_ROWS || n_real > PF_ROWS || k < 1) return cudaErrorInvalidValue;
    k_prune_floor<<<1, PF_ROWS, 0, st>>>(bound, n_real, lb, lb_rows, order, n_lb_rows, k,
                                         floor_out);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ launchers
template <bool SIGNED>
static cudaError_t launch_kth(const SelectPlan &sp, const float *s, int b, const int32_t *ext_of,
                              int64_t id_limit, unsigned long long *ws, unsigned long long *bound,
                              unsigned int *cnt, cudaStream_t st, uint32_t slack = 0,
                              NsScope ns = NsScope{}) {
    static bool attr[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr[dev]) {
        cudaError_t e = cudaFuncSetAttribute(k_sample_kth,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             KTH_STAGE * (int)sizeof(uint32_t));
        if (e != cudaSuccess) return e;
        attr[dev] = true;
    }
    uint32_t *keysT = (uint32_t *)(ws + sp.off_tr);
    const dim3 tgrid((unsigned)ceil_div<int64_t>(sp.n_sample, 32), (unsigned)(sp.bp / 32));
    k_sample_transpose<SIGNED><<<tgrid, 256, 0, st>>>(s, sp.n_sample, sp.stride, sp.bp, ext_of,
                                                      id_limit, ns, keysT);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const size_t smem = sp.n_sample <= KTH_STAGE ? (size_t)sp.n_sample * sizeof(uint32_t) : 0;
    k_sample_kth<<<sp.bp, SEL_THREADS, smem, st>>>(keysT, sp.n_sample, b, sp.k, slack, bound,
                                                   cnt);
    return cudaGetLastError();
}

template <bool SIGNED>
static cudaError_t bound_and_filter(const SelectPlan &sp, const float *s, int b,
                                    const int32_t *ext_of, int64_t id_limit,
                                    unsigned long long *ws, cudaStream_t st, int *launches,
                                    NsScope ns = NsScope{}) {
    unsigned long long *bound = ws + sp.off_bound;
    unsigned int *cnt = (unsigned int *)(ws + sp.off_cnt);
    unsigned long long *buf = ws + sp.off_buf;
    cudaError_t e = launch_kth<SIGNED>(sp, s, b, ext_of, id_limit, ws, bound, cnt, st, 0, ns);
    if (e != cudaSuccess) return e;
    const int64_t warps = ceil_div<int64_t>(sp.n, 4);
    int grid = (int)(ceil_div<int64_t>(warps, 8) < (int64_t)device_sm_count() * 8
                         ? ceil_div<int64_t>(warps, 8)
                         : (int64_t)device_sm_count() * 8);
    grid = grid < 1 ? 1 : grid;
    switch (sp.bp) {
    case 32: k_filter<32, SIGNED><<<grid, 256, 0, st>>>(s, sp.n, ext_of, id_limit, ns, bound, cnt, buf, sp.cap); break;
    case 64: k_filter<64, SIGNED><<<grid, 256, 0, st>>>(s, sp.n, ext_of, id_limit, ns, bound, cnt, buf, sp.cap); break;
    case 128: k_filter<128, SIGNED><<<grid, 256, 0, st>>>(s, sp.n, ext_of, id_limit, ns, bound, cnt, buf, sp.cap); break;
    case 256: k_filter<256, SIGNED><<<grid, 256, 0, st>>>(s, sp.n, ext_of, id_limit, ns, bound, cnt, buf, sp.cap); break;
    default: return cudaErrorInvalidValue;
    }
    if (launches) *launches += 3;
    return cudaGetLastError();
}

template <bool SIGNED>
static cudaError_t sample_bound(const SelectPlan &sp, const float *s, int b,
                                const int32_t *ext_of, int64_t id_limit,
                                unsigned long long *ws, unsigned long long *bound,
                                cudaStream_t st, int *launches, uint32_t slack = 0,
                                NsScope ns = NsScope{}) {
    cudaError_t e = launch_kth<SIGNED>(sp, s, b, ext_of, id_limit, ws, bound,
                                       (unsigned int *)(ws + sp.off_cnt), st, slack, ns);
    if (launches) *launches += 2;
    return e;
}

cudaError_t launch_sample_bound_signed(const SelectPlan &sp, const float *s, int b,
                                       const int32_t *ext_of, int64_t id_limit,
                                       unsigned long long *ws, unsigned long long *bound,
                                       cudaStream_t st, int *launches, NsScope ns) {
    return sample_bound<true>(sp, s, b, ext_of, id_limit, ws, bound, st, launches, 0, ns);
}

cudaError_t launch_sample_bound(const SelectPlan &sp, const float *s, int b,
                                const int32_t *ext_of, unsigned long long *ws, cudaStream_t st,
                                int *launches, uint32_t slack, NsScope ns) {
    return sample_bound<false>(sp, s, b, ext_of, (int64_t)1 << 40, ws, ws + sp.off_bound, st,
                               launches, slack, ns);
}

cudaError_t launch_select(const SelectPlan &sp, const float *s, int b, unsigned long long *ws,
                          const float *zpart, int64_t n_ztiles, const int32_t *ext_of,
                          const int32_t *row_of, const int32_t *page_row, int64_t *ids,
                          float *scores, int32_t *page_ids, int32_t *n_pages, int *status,
                          NsScope ns, int sort_by_time, cudaStream_t st, int *launches) {
    cudaError_t e = bound_and_filter<false>(sp, s, b, ext_of, (int64_t)1 << 40, ws, st, launches,
                                            ns);
    if (e != cudaSuccess) return e;
    return launch_topk_merge(sp, s, b, ws, zpart, n_ztiles, ext_of, row_of, page_row, ids, scores,
                             page_ids, n_pages, status, nullptr, ns, sort_by_time, st, launches);
}

cudaError_t launch_topk_merge(const SelectPlan &sp, const float *s, int b,
                              const unsigned long long *ws, const float *zpart, int64_t n_ztiles,
                              const int32_t *ext_of, const int32_t *row_of,
                              const int32_t *page_row, int64_t *ids, float *scores,
                              int32_t *page_ids, int32_t *n_pages, int *status,
                              const ColumnRecompute *rc, NsScope ns, int sort_by_time,
                              cudaStream_t st, int *launches) {
    ColumnRecompute r{};
    if (rc) r = *rc;
    cudaError_t e = launch_pdl(k_topk_merge, dim3(b), dim3(SEL_THREADS), 0, st, s, sp.n, sp.bp,
                               sp.k, ext_of, (const unsigned int *)(ws + sp.off_cnt),
                               (const unsigned long long *)(ws + sp.off_buf), sp.cap, zpart,
                               n_ztiles, row_of, page_row, ids, scores, page_ids, n_pages, status,
                               r, ns, sort_by_time);
    if (launches) *launches += 1;
    return e == cudaSuccess ? cudaGetLastError() : e;
}

cudaError_t launch_select_signed(const SelectPlan &sp, const float *s, int b,
                                 unsigned long long *ws, const int32_t *ext_of, int64_t id_limit,
                                 int64_t c_base, int32_t *nbr_ids, float *nbr_cos, int *status,
                                 cudaStream_t st, int *launches, NsScope ns) {
    cudaError_t e = bound_and_filter<true>(sp, s, b, ext_of, id_limit, ws, st, launches, ns);
    if (e != cudaSuccess) return e;
    k_topm_merge<<<b, SEL_THREADS, 0, st>>>(s, sp.n, sp.bp, sp.k, ext_of, id_limit,
                                            (const unsigned int *)(ws + sp.off_cnt),
                                            ws + sp.off_buf, sp.cap, c_base, nbr_ids, nbr_cos,
                                            status, ns);
    if (launches) *launches += 1;
    return cudaGetLastError();
}

}  // namespace ak
