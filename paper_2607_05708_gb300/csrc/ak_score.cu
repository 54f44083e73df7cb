// Score step (a1) of query-aware retrieval: z = tau * E q^T, u = exp(z - c),
// with per-tile partial sums toward Z = sum_i u (arXiv 2607.05708, §4.1,
// Dense-only form of §5.5).  Also the query preparation and the running
// maximum of chunk-embedding norms used for the shift bound c.
#include "ak_common.cuh"

namespace ak {

// ------------------------------------------------------------------ query prep
// One CTA per padded query row.  shift[c] = tau * |q_c| * max_i |e_i| bounds
// z from above, so u = exp(z - shift) <= 1 never overflows; padding rows are
// zero with shift 0.
__global__ void k_prep_queries(const uint16_t *__restrict__ q, int b, int dim, float tau,
                               const float *__restrict__ max_norm, uint16_t *__restrict__ qp,
                               float *__restrict__ shift, int *status) {
    const int c = blockIdx.x;
    __shared__ float red[32];
    float ss = 0.f;
    for (int t = threadIdx.x; t < dim; t += blockDim.x) {
        uint16_t h = (c < b) ? q[(int64_t)c * dim + t] : (uint16_t)0;
        qp[(int64_t)c * dim + t] = h;
        float v = bf16_to_f32(h);
        ss = fmaf(v, v, ss);
    }
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    if (threadIdx.x == 0) {
        float tot = 0.f;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += red[w];
        float s = (c < b) ? tau * sqrtf(tot) * (*max_norm) : 0.f;
        shift[c] = s;
        if (!(2.f * s <= 80.f)) set_status(status, AKASHIC_ERANGE);
    }
}

cudaError_t launch_prep_queries(const uint16_t *q, int b, int bp, int dim, float tau,
                                const float *max_norm, uint16_t *qp, float *shift, int *status,
                                cudaStream_t st) {
    k_prep_queries<<<bp, 128, 0, st>>>(q, b, dim, tau, max_norm, qp, shift, status);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ norm max
// One warp per row; the running maximum only grows (appends never shrink it).
__global__ void k_row_norm_max(const uint16_t *__restrict__ emb, int64_t n, int dim,
                               float *max_norm) {
    const int lane = threadIdx.x & 31;
    int64_t row = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t stride = ((int64_t)gridDim.x * blockDim.x) >> 5;
    float best = 0.f;
    for (; row < n; row += stride) {
        const uint16_t *e = emb + row * dim;
        float ss = 0.f;
        for (int t = lane; t < dim; t += 32) {
            float v = bf16_to_f32(e[t]);
            ss = fmaf(v, v, ss);
        }
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        best = fmaxf(best, sqrtf(ss));
    }
    if (lane == 0) atomicMax((int *)max_norm, __float_as_int(best));   // non-negative floats
}

cudaError_t launch_row_norm_max(const uint16_t *emb, int64_t n, int dim, float *max_norm,
                                cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    int64_t warps = n < (int64_t)152 * 64 ? n : (int64_t)152 * 64;
    int grid = (int)ceil_div<int64_t>(warps * 32, 256);
    k_row_norm_max<<<grid, 256, 0, st>>>(emb, n, dim, max_norm);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ score GEMM
// Tiled SIMT GEMM: a 64-row x 64-query tile per CTA, K in steps of 32,
// each thread a 4 x 4 block of outputs, fp32 accumulation of exactly
// widened bf16 values.  The epilogue applies exp(tau*acc - shift) and sums
// each query column over the tile's rows.
constexpr int SM_TM = 64, SM_TN = 64, SM_TK = 32;

int64_t score_tiles(int64_t n) { return ceil_div<int64_t>(n, SM_TM); }

template <bool EXP>
__global__ __launch_bounds__(256) void k_score_simt(const uint16_t *__restrict__ emb, int64_t n,
                                                    int dim, const uint16_t *__restrict__ qp,
                                                    int bp, const float *__restrict__ shift,
                                                    float tau, float *__restrict__ u,
                                                    float *__restrict__ zpart) {
    __shared__ float As[SM_TK][SM_TM + 4];
    __shared__ float Bs[SM_TK][SM_TN + 4];
    __shared__ float zs[16][SM_TN];
    const int64_t tile = blockIdx.x;
    const int64_t r0 = tile * SM_TM;
    const int c0 = blockIdx.y * SM_TN;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

    for (int k0 = 0; k0 < dim; k0 += SM_TK) {
        for (int i = threadIdx.x; i < SM_TM * SM_TK; i += 256) {
            int r = i / SM_TK, kk = i % SM_TK;
            int64_t row = r0 + r;
            As[kk][r] = row < n ? bf16_to_f32(emb[row * dim + k0 + kk]) : 0.f;
        }
        for (int i = threadIdx.x; i < SM_TN * SM_TK; i += 256) {
            int c = i / SM_TK, kk = i % SM_TK;
            int col = c0 + c;
            Bs[kk][c] = col < bp ? bf16_to_f32(qp[(int64_t)col * dim + k0 + kk]) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < SM_TK; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
    float colsum[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        int64_t row = r0 + ty * 4 + i;
        if (row >= n) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            int col = c0 + tx * 4 + j;
            if (col < bp) {
                float v = EXP ? expf(tau * acc[i][j] - shift[col]) : acc[i][j];
                u[row * bp + col] = v;
                colsum[j] += v;
            }
        }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) zs[ty][tx * 4 + j] = colsum[j];
    if (!EXP) return;
    __syncthreads();
    if (threadIdx.x < SM_TN) {
        int col = c0 + threadIdx.x;
        if (col < bp) {
            float s = 0.f;
#pragma unroll
            for (int r = 0; r < 16; ++r) s += zs[r][threadIdx.x];
            zpart[tile * bp + col] = s;
        }
    }
}

cudaError_t launch_score(const uint16_t *emb, int64_t n, int dim, const uint16_t *qp, int bp,
                         const float *shift, float tau, float *u, float *zpart, int *status,
                         cudaStream_t st, int *launches) {
    (void)status;
    dim3 grid((unsigned)score_tiles(n), (unsigned)ceil_div(bp, SM_TN));
    k_score_simt<true><<<grid, 256, 0, st>>>(emb, n, dim, qp, bp, shift, tau, u, zpart);
    if (launches) *launches += 1;
    return cudaGetLastError();
}

cudaError_t launch_dots(const uint16_t *emb, int64_t n, int dim, const uint16_t *qp, int bp,
                        float *out, cudaStream_t st, int *launches) {
    dim3 grid((unsigned)score_tiles(n), (unsigned)ceil_div(bp, SM_TN));
    k_score_simt<false><<<grid, 256, 0, st>>>(emb, n, dim, qp, bp, nullptr, 1.f, out, nullptr);
    if (launches) *launches += 1;
    return cudaGetLastError();
}

}  // namespace ak
