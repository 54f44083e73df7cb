// Two-hop scores of the top-k candidates without the hops.
//
// Unrolling the hop recursion s^(h) = u + alpha R^T s^(h-1) (the relation
// propagation of §4.1, R_ki = w(k -> i)) gives, for a row j,
//   s^(H)_j = u_j + sum_{t=1..H} alpha^t sum_k C_t[k][j] u_k,
//   C_1[k][j] = w(k -> j),   C_t = R C_{t-1},
// with reach coefficients C_t that depend on the graph alone.  The row
// bounds of the last hop (ak_graph.cu) prove that only the rows whose
// upper bound reaches the top-k floor can be selected; when all of them lie
// in a small set of heavy candidate rows whose coefficients are kept, their
// final scores for every query come from one pass over the score slab u,
// and the hops are not run.  The selection is the same as the hops' (the
// values differ only by fp32 summation order).
#include "ak_common.cuh"

namespace ak {

// ------------------------------------------------------------------ graph-only
// Candidates: the REACH_T rows of largest upper mass sum_{t<=H} mup[t]
// among the (up to 1024) heaviest split rows; ties to the lower row.  One
// CTA of 1024 threads, bitonic sort of the keys in shared memory.
__global__ __launch_bounds__(1024) void k_reach_pick(const int32_t *__restrict__ split_row,
                                                      const int32_t *__restrict__ split_order,
                                                      int64_t n_split,
                                                      const float *__restrict__ mup, int64_t n,
                                                      int H, int32_t *__restrict__ rows,
                                                      int *__restrict__ t_out) {
    __shared__ unsigned long long key[1024];
    const int tid = threadIdx.x;
    const int nc = (int)(n_split < 1024 ? n_split : 1024);
    unsigned long long k = 0ull;
    if (tid < nc) {
        const int32_t r = split_row[split_order[tid]];
        float m = 0.f;
        for (int t = 1; t <= H; ++t) m += mup[(int64_t)t * n + r];
        k = ((unsigned long long)__float_as_uint(m) << 32) | (unsigned long long)(~(uint32_t)r);
    }
    key[tid] = k;
    __syncthreads();
    // descending bitonic sort
    for (int size = 2; size <= 1024; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const int other = tid ^ stride;
            if (other > tid) {
                const unsigned long long a = key[tid], b = key[other];
                const bool desc = (tid & size) == 0;
                if (desc ? a < b : a > b) {
                    key[tid] = b;
                    key[other] = a;
                }
            }
            __syncthreads();
        }
    }
    const int T = nc < REACH_T ? nc : REACH_T;
    if (tid < T) rows[tid] = (int32_t)~(uint32_t)(key[tid] & 0xffffffffull);
    if (tid == 0) *t_out = T;
}

__global__ void k_reach_map(const int32_t *__restrict__ rows, const int *__restrict__ t_cnt,
                            int32_t *__restrict__ map) {
    if ((int)threadIdx.x < *t_cnt) map[rows[threadIdx.x]] = (int32_t)threadIdx.x;
}

// C_1[k][t] = w(k -> rows[t]): the candidate's in-edges (one CTA each).
__global__ void k_reach_c1(const int32_t *__restrict__ rows, const int *__restrict__ t_cnt,
                           const int64_t *__restrict__ in_ptr, const int32_t *__restrict__ in_src,
                           const float *__restrict__ in_w, float *__restrict__ C1) {
    const int t = blockIdx.x;
    if (t >= *t_cnt) return;
    const int64_t j = rows[t];
    for (int64_t e = in_ptr[j] + threadIdx.x; e < in_ptr[j + 1]; e += blockDim.x)
        C1[(int64_t)in_src[e] * REACH_T + t] = in_w[e];
}

// Cn[row(k)][:] = sum over k's out-edges (k -> i) of w * Cp[row(i)][:]: one
// warp per chunk ID k, four columns per lane (a float4), edges in CSR order.
__global__ void k_reach_spmm(const int64_t *__restrict__ row_ptr, const int32_t *__restrict__ col,
                             const float *__restrict__ w, const int32_t *__restrict__ row_of,
                             int64_t n, const float *__restrict__ Cp, float *__restrict__ Cn) {
    static_assert(REACH_T == 128, "four columns per lane");
    const int lane = threadIdx.x & 31;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t k = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; k < n; k += nw) {
        float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int64_t e = row_ptr[k]; e < row_ptr[k + 1]; ++e) {
            const float we = w[e];
            const float4 c =
                reinterpret_cast<const float4 *>(Cp + (int64_t)row_of[col[e]] * REACH_T)[lane];
            a.x = fmaf(we, c.x, a.x);
            a.y = fmaf(we, c.y, a.y);
            a.z = fmaf(we, c.z, a.z);
            a.w = fmaf(we, c.w, a.w);
        }
        reinterpret_cast<float4 *>(Cn + (int64_t)row_of[k] * REACH_T)[lane] = a;
    }
}

cudaError_t launch_reach_build(const ReachBuild &rb, cudaStream_t st) {
    const int sms = device_sm_count();
    cudaError_t e = cudaMemsetAsync(rb.map, 0xff, (size_t)rb.n * 4, st);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(rb.C, 0, (size_t)rb.H * rb.n * REACH_T * 4, st);
    if (e != cudaSuccess) return e;
    k_reach_pick<<<1, 1024, 0, st>>>(rb.split_row, rb.split_order, rb.n_split, rb.mup, rb.n, rb.H,
                                     rb.rows, rb.t_cnt);
    k_reach_map<<<1, REACH_T, 0, st>>>(rb.rows, rb.t_cnt, rb.map);
    k_reach_c1<<<REACH_T, 256, 0, st>>>(rb.rows, rb.t_cnt, rb.in_ptr, rb.in_src, rb.in_w, rb.C);
    for (int t = 2; t <= rb.H; ++t)
        k_reach_spmm<<<sms * 8, 256, 0, st>>>(rb.row_ptr, rb.col, rb.w, rb.row_of, rb.n,
                                              rb.C + (int64_t)(t - 2) * rb.n * REACH_T,
                                              rb.C + (int64_t)(t - 1) * rb.n * REACH_T);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ per call
// Rows whose upper bound reaches the floor: a candidate's slot is flagged,
// any other row counted in *bad (then the hops run instead).
__global__ void k_reach_check(const float *__restrict__ ub, const float *__restrict__ floor_p,
                              const int32_t *__restrict__ map, int64_t n,
                              int32_t *__restrict__ keep, int *__restrict__ bad) {
    const float floor_ = *floor_p;
    int nb = 0;
    for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n;
         j += (int64_t)gridDim.x * blockDim.x) {
        if (ub[j] >= floor_) {
            const int32_t t = map[j];
            if (t >= 0) keep[t] = 1;
            else ++nb;
        }
    }
    if (nb) atomicAdd(bad, nb);
}

// The flagged candidates' combined coefficients, contiguous:
// coefK[k][i] = sum_t alpha^t C_t[k][slot_i] for i < nk, 0 up to NK8.
__global__ void k_reach_coef(const float *__restrict__ C, int64_t n, int H, float alpha,
                             const ReachSlots rs, int nk8, float *__restrict__ coefK) {
    for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < n * nk8;
         x += (int64_t)gridDim.x * blockDim.x) {
        const int64_t k = x / nk8;
        const int i = (int)(x - k * nk8);
        float c = 0.f;
        if (i < rs.nk) {
            const int64_t at = k * REACH_T + rs.slot[i];
            for (int t = H; t >= 1; --t) c = alpha * (c + C[(int64_t)(t - 1) * n * REACH_T + at]);
        }
        coefK[x] = c;
    }
}

__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                     (uint32_t)__cvta_generic_to_shared(dst)),
                 "l"(src)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// partial[cta][i][b] = sum over this CTA's rows k of coefK[k][i] u[k][b]
// (BP = 256 or 128 columns of u).  REACH_T_THREADS threads: thread t takes
// columns 4 (t % (BP/4)) + 0..3 and one of G = 512 / BP slot groups
// (t / (BP/4)), so that one shared load of four coefficients feeds sixteen
// FMAs; REACH_ROWS rows at a time are copied to shared memory (u rows and
// coefficient rows) with cp.async, double-buffered so that the next rows
// load while these are summed; rows in order.
constexpr int REACH_ROWS = 32;
constexpr int REACH_T_THREADS = 128;

template <int NK, int BP>
__global__ __launch_bounds__(REACH_T_THREADS, 2) void k_reach_terms(
    const float *__restrict__ u, int64_t n, const float *__restrict__ coefK, int nk,
    float *__restrict__ partial) {
    extern __shared__ __align__(16) float dyn[];
    constexpr int TT = REACH_T_THREADS;
    constexpr int G = TT / (BP / 4);                   // slot groups (= 512 / BP)
    constexpr int HALF = NK / G;                       // slots per thread
    static_assert(G * (BP / 4) == TT, "every thread one column quad and one slot group");
    static_assert(HALF % 4 == 0, "four coefficients per shared load");
    float *us = dyn;                                   // [2][REACH_ROWS][BP]
    float *cs = dyn + 2 * REACH_ROWS * BP;             // [2][REACH_ROWS][NK]
    const int cg = threadIdx.x % (BP / 4), sg = threadIdx.x / (BP / 4);
    const int64_t per = (n + gridDim.x - 1) / gridDim.x;
    const int64_t k0 = (int64_t)blockIdx.x * per;
    const int64_t k1 = k0 + per < n ? k0 + per : n;
    const int64_t n_chunks = (k1 - k0 + REACH_ROWS - 1) / REACH_ROWS;
    auto stage = [&](int64_t c, int buf) {
        const int64_t kb = k0 + c * REACH_ROWS;
        const int rows = (int)(k1 - kb < REACH_ROWS ? k1 - kb : REACH_ROWS);
        float *ud = us + buf * REACH_ROWS * BP;
        float *cd = cs + buf * REACH_ROWS * NK;
        // u rows: rows x BP/4 pieces of 16 bytes; coefficient rows: rows x NK/4
        for (int x = threadIdx.x; x < rows * (BP / 4); x += TT)
            cp_async16(ud + x * 4, u + kb * BP + (int64_t)x * 4);
        for (int x = threadIdx.x; x < rows * (NK / 4); x += TT)
            cp_async16(cd + x * 4, coefK + kb * NK + (int64_t)x * 4);
        cp_async_commit();
    };
    float acc[HALF][4];
#pragma unroll
    for (int i = 0; i < HALF; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
    if (n_chunks > 0) stage(0, 0);
    for (int64_t c = 0; c < n_chunks; ++c) {
        const int buf = (int)(c & 1);
        if (c + 1 < n_chunks) {
            stage(c + 1, buf ^ 1);
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        const int64_t kb = k0 + c * REACH_ROWS;
        const int rows = (int)(k1 - kb < REACH_ROWS ? k1 - kb : REACH_ROWS);
        const float *ud = us + buf * REACH_ROWS * BP;
        const float *cd = cs + buf * REACH_ROWS * NK;
#pragma unroll 2
        for (int r = 0; r < rows; ++r) {
            const float4 x = *reinterpret_cast<const float4 *>(ud + r * BP + 4 * cg);
            const float4 *c4 = reinterpret_cast<const float4 *>(cd + r * NK + sg * HALF);
#pragma unroll
            for (int q = 0; q < HALF / 4; ++q) {
                const float4 cq = c4[q];
                const float cv[4] = {cq.x, cq.y, cq.z, cq.w};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    acc[4 * q + i][0] = fmaf(cv[i], x.x, acc[4 * q + i][0]);
                    acc[4 * q + i][1] = fmaf(cv[i], x.y, acc[4 * q + i][1]);
                    acc[4 * q + i][2] = fmaf(cv[i], x.z, acc[4 * q + i][2]);
                    acc[4 * q + i][3] = fmaf(cv[i], x.w, acc[4 * q + i][3]);
                }
            }
        }
        __syncthreads();   // this buffer is restaged two chunks later
    }
#pragma unroll
    for (int i = 0; i < HALF; ++i) {
        const int slot = sg * HALF + i;
        if (slot < nk)
            *reinterpret_cast<float4 *>(partial + ((int64_t)blockIdx.x * REACH_T + slot) * BP +
                                        4 * cg) =
                make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
    }
}

// Final score of each flagged candidate for each real query column: its u
// plus the CTAs' partials, appended as a filter key (score bits, ~chunk ID)
// to the column's buffer; the buffer then holds exactly them.  One block per
// candidate: thread t takes column t % bp and every (1024 / bp)-th partial
// from t / bp on (coalesced rows of the partials), and the groups are added
// in group order (the same order on every run).
__global__ __launch_bounds__(1024) void k_reach_emit(const float *__restrict__ u, int bp, int B,
                                                     const float *__restrict__ partial,
                                                     int n_parts, const ReachSlots rs,
                                                     const int32_t *__restrict__ rows,
                                                     const int32_t *__restrict__ ext_of,
                                                     unsigned int *__restrict__ cnt,
                                                     unsigned long long *__restrict__ buf,
                                                     int64_t cap) {
    __shared__ float red[1024];
    const int i = blockIdx.x;
    const int b = threadIdx.x % bp, g = threadIdx.x / bp, ng = blockDim.x / bp;
    float acc = 0.f;
#pragma unroll 16
    for (int p = g; p < n_parts; p += ng) acc += partial[((int64_t)p * REACH_T + i) * bp + b];
    red[threadIdx.x] = acc;
    __syncthreads();
    if (g == 0 && b < B) {
        float sum = red[b];
        for (int h = 1; h < ng; ++h) sum += red[h * bp + b];
        const int64_t j = rows[rs.slot[i]];
        const float s = u[j * bp + b] + sum;
        buf[(int64_t)b * cap + i] = ((unsigned long long)__float_as_uint(s) << 32) |
                                    (unsigned long long)(~(uint32_t)ext_of[j]);
        if (i == 0) cnt[b] = (unsigned int)rs.nk;
    }
}

cudaError_t launch_reach_check(const float *ub, const float *floor_p, const int32_t *map,
                               int64_t n, int32_t *keep, int *bad, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(keep, 0, REACH_T * 4, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(bad, 0, 4, st);
    if (e != cudaSuccess) return e;
    k_reach_check<<<device_sm_count() * 4, 256, 0, st>>>(ub, floor_p, map, n, keep, bad);
    return cudaGetLastError();
}

int reach_parts() { return device_sm_count() * 2; }

// The packed width: the flagged count rounded up to 8 (bp = 256) or 16.
static int reach_width(int bp, int nk) { return bp == 256 ? (nk + 7) & ~7 : (nk + 15) & ~15; }

size_t reach_coef_floats(int64_t n, int bp, int nk) { return (size_t)n * reach_width(bp, nk); }

cudaError_t launch_reach_coef(const float *C, int64_t n, int H, float alpha, const ReachSlots &rs,
                              int bp, float *coefK, cudaStream_t st) {
    const int nk8 = reach_width(bp, rs.nk);
    k_reach_coef<<<device_sm_count() * 8, 256, 0, st>>>(C, n, H, alpha, rs, nk8, coefK);
    return cudaGetLastError();
}

template <int NK, int BP>
static cudaError_t reach_terms_nk(const float *u, int64_t n, const float *coefK, int nk,
                                  float *partial, int parts, cudaStream_t st) {
    const size_t smem = (size_t)2 * REACH_ROWS * (BP + NK) * sizeof(float);
    static bool attr[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr[dev]) {
        cudaError_t e = cudaFuncSetAttribute(k_reach_terms<NK, BP>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr[dev] = true;
    }
    k_reach_terms<NK, BP><<<parts, REACH_T_THREADS, smem, st>>>(u, n, coefK, nk, partial);
    return cudaGetLastError();
}

// Flagged counts the score pass takes: NK (rounded up to 8 / 16) at most 64
// slots per thread group pair at BP = 256, 128 at BP = 128.
bool reach_fits(int bp, int nk) {
    return nk >= 1 && ((bp == 256 && nk <= 64) || (bp == 128 && nk <= 128));
}

cudaError_t launch_reach_scores(const float *u, int bp, int B, int64_t n, const float *coefK,
                                const ReachSlots &rs, const int32_t *rows, const int32_t *ext_of,
                                float *partial, unsigned int *cnt, unsigned long long *buf,
                                int64_t cap, cudaStream_t st, int *launches) {
    if (!reach_fits(bp, rs.nk)) return cudaErrorInvalidValue;
    const int parts = reach_parts();
    cudaError_t e = cudaErrorInvalidValue;
    if (bp == 256) {
        switch ((rs.nk + 7) & ~7) {
        case 8: e = reach_terms_nk<8, 256>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 16: e = reach_terms_nk<16, 256>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 24: e = reach_terms_nk<24, 256>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 32: e = reach_terms_nk<32, 256>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 40: e = reach_terms_nk<40, 256>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 48: e = reach_terms_nk<48, 256>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 56: e = reach_terms_nk<56, 256>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 64: e = reach_terms_nk<64, 256>(u, n, coefK, rs.nk, partial, parts, st); break;
        default: break;
        }
    } else {
        switch ((rs.nk + 15) & ~15) {
        case 16: e = reach_terms_nk<16, 128>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 32: e = reach_terms_nk<32, 128>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 48: e = reach_terms_nk<48, 128>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 64: e = reach_terms_nk<64, 128>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 80: e = reach_terms_nk<80, 128>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 96: e = reach_terms_nk<96, 128>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 112: e = reach_terms_nk<112, 128>(u, n, coefK, rs.nk, partial, parts, st); break;
        case 128: e = reach_terms_nk<128, 128>(u, n, coefK, rs.nk, partial, parts, st); break;
        default: break;
        }
    }
    if (e != cudaSuccess) return e;
    k_reach_emit<<<rs.nk, 1024, 0, st>>>(u, bp, B, partial, parts, rs, rows, ext_of, cnt, buf, cap);
    if (launches) *launches += 2;
    return cudaGetLastError();
}

}  // namespace ak
