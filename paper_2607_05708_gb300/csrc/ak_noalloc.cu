// Softmax scores without any device allocation.
//
// Some callers cannot allocate device memory at the moment they need the
// scores: code recording work into a CUDA graph or running inside a
// pre-reserved memory pool of a serving runtime must not call cudaMalloc
// (it would synchronise the device or break the capture), and embedded
// hosts may have no allocator at all.  For them this file offers one entry
// point that computes the score step of retrieval over caller-owned buffers
// and keeps its own scratch in a fixed, file-scope device array.
//
// Scratch: NOALLOC_SCRATCH_BYTES (320 KiB) in `g_noalloc_scratch`, holding
// the running norm bound, the per-query shifts, a status word and one row
// of partial sums per CTA of the score kernel (at most NOALLOC_MAX_CTAS).
// Every GPU on which this entry point runs holds that array until the
// process exits.  All calls share it: two calls whose work overlaps on the
// GPU (different streams, no ordering between them) race on it.
#include <stdarg.h>
#include <stdio.h>

#include <mutex>

#include "ak_common.cuh"

namespace ak {

constexpr size_t NOALLOC_SCRATCH_BYTES = 320 * 1024;
constexpr int NOALLOC_MAX_B = 256;
constexpr int NOALLOC_MAX_CTAS = 256;
// byte offsets inside the scratch array
constexpr size_t NA_NORM = 0;       // float: max row norm of the embeddings
constexpr size_t NA_STATUS = 64;    // int: device status word
constexpr size_t NA_SHIFT = 256;    // float[NOALLOC_MAX_B]
constexpr size_t NA_ZPART = 2048;   // float[NOALLOC_MAX_CTAS][NOALLOC_MAX_B]
static_assert(NA_ZPART + (size_t)NOALLOC_MAX_CTAS * NOALLOC_MAX_B * 4 <= NOALLOC_SCRATCH_BYTES,
              "scratch layout exceeds the array");

static __device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_SCRATCH_BYTES];

// Clear the values that must start at zero (norm bound, status).
__global__ void k_noalloc_reset(unsigned char *scratch) {
    if (threadIdx.x == 0) {
        *(float *)(scratch + NA_NORM) = 0.f;
        *(int *)(scratch + NA_STATUS) = 0;
    }
}

// shift[c] = tau * |q_c| * max_j |e_j| (one CTA per query row).
__global__ void k_noalloc_shift(const uint16_t *__restrict__ q, int dim, float tau,
                                unsigned char *scratch) {
    const int c = blockIdx.x;
    __shared__ float red[32];
    float ss = 0.f;
    for (int t = threadIdx.x; t < dim; t += blockDim.x) {
        const float v = bf16_to_f32(q[(int64_t)c * dim + t]);
        ss = fmaf(v, v, ss);
    }
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    if (threadIdx.x == 0) {
        float tot = 0.f;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += red[w];
        const float s = tau * sqrtf(tot) * *(const float *)(scratch + NA_NORM);
        ((float *)(scratch + NA_SHIFT))[c] = s;
        if (!(2.f * s <= 80.f)) set_status((int *)(scratch + NA_STATUS), AKASHIC_ERANGE);
    }
}

// z[c] = sum of the score kernel's partial sums; optional copies of the
// shifts and of the status word (cleared again by the next call's reset).
__global__ void k_noalloc_finish(const unsigned char *scratch, int b, int zrows, float *z,
                                 float *shift_out, int32_t *status_out) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c < b) {
        const float *zp = (const float *)(scratch + NA_ZPART);
        double acc = 0.0;
        for (int r = 0; r < zrows; ++r) acc += (double)zp[(int64_t)r * b + c];
        z[c] = (float)acc;
        if (shift_out) shift_out[c] = ((const float *)(scratch + NA_SHIFT))[c];
    }
    if (c == 0 && status_out) *status_out = *(const int *)(scratch + NA_STATUS);
}

static akashic_status_t noalloc_fail(akashic_status_t code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    set_last_error(buf);
    return code;
}

// Set-up on the first call made on a device (with that device current):
// the device address of the scratch array, and the score kernel's
// shared-memory limit for all four query widths, so that later calls with
// any B do no set-up at all.
static std::mutex g_noalloc_mu;
static unsigned char *g_noalloc_ptr[64] = {nullptr};

static cudaError_t noalloc_scratch(int dev, unsigned char **out) {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void *p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e == cudaSuccess) e = prepare_score_gemm();
        if (e != cudaSuccess) return e;
        g_noalloc_ptr[dev] = (unsigned char *)p;
    }
    *out = g_noalloc_ptr[dev];
    return cudaSuccess;
}

}  // namespace ak

using namespace ak;

extern "C" akashic_status_t akashic_mem_softmax_scores_noalloc(const uint16_t *emb, int64_t n,
                                                           int32_t dim, const uint16_t *q,
                                                           int32_t B, float temperature, float *u,
                                                           float *z, float *shift,
                                                           int32_t *status, void *stream) {
    set_last_error("");
    if (!emb || !q || !u || !z) return noalloc_fail(AKASHIC_EINVAL, "softmax_scores_noalloc: NULL argument");
    if (n < 1 || n > 0x7fffffffLL) return noalloc_fail(AKASHIC_EINVAL, "softmax_scores_noalloc: n must be in [1, 2^31-1]");
    if (dim < 64 || dim > 4096 || dim % 64 != 0)
        return noalloc_fail(AKASHIC_EINVAL, "softmax_scores_noalloc: dim must be a multiple of 64 in [64, 4096]");
    if (B != 32 && B != 64 && B != 128 && B != 256)
        return noalloc_fail(AKASHIC_EINVAL,
                            "softmax_scores_noalloc: B must be 32, 64, 128 or 256 (at most %d queries "
                            "fit the fixed scratch)", NOALLOC_MAX_B);
    if (!(temperature >= 0.f) || !isfinite(temperature))
        return noalloc_fail(AKASHIC_EINVAL, "softmax_scores_noalloc: temperature must be finite and >= 0");
    if (((uintptr_t)emb | (uintptr_t)q | (uintptr_t)u) & 15u)
        return noalloc_fail(AKASHIC_EINVAL, "softmax_scores_noalloc: emb, q and u must be 16-byte aligned");
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        cudaGetLastError();
        return noalloc_fail(AKASHIC_ECUDA, "softmax_scores_noalloc: no current CUDA device");
    }
    if (device_sm_count() > NOALLOC_MAX_CTAS)
        return noalloc_fail(AKASHIC_EINVAL,
                            "softmax_scores_noalloc: %d SMs exceed the %d partial-sum rows of the "
                            "fixed scratch", device_sm_count(), NOALLOC_MAX_CTAS);
    unsigned char *scr = nullptr;
    cudaError_t e = noalloc_scratch(dev, &scr);
    if (e != cudaSuccess)
        return noalloc_fail(AKASHIC_ECUDA, "softmax_scores_noalloc: set-up on this device: %s",
                            cudaGetErrorString(e));
    cudaStream_t st = (cudaStream_t)stream;
    const float tau = temperature > 0.f ? temperature : 1.0f / sqrtf((float)dim);
    k_noalloc_reset<<<1, 32, 0, st>>>(scr);
    e = cudaGetLastError();
    if (e == cudaSuccess) e = launch_row_norm_max(emb, n, dim, (float *)(scr + NA_NORM), st);
    if (e == cudaSuccess) {
        k_noalloc_shift<<<B, 128, 0, st>>>(q, dim, tau, scr);
        e = cudaGetLastError();
    }
    int zrows = 0;
    if (e == cudaSuccess)
        e = launch_score(emb, n, dim, q, B, (const float *)(scr + NA_SHIFT), tau, u,
                         (float *)(scr + NA_ZPART), (int *)(scr + NA_STATUS), st, nullptr, &zrows);
    if (e == cudaSuccess) {
        k_noalloc_finish<<<ceil_div(B, 256), 256, 0, st>>>(scr, B, zrows, z, shift, status);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess)
        return noalloc_fail(AKASHIC_ECUDA, "softmax_scores_noalloc: launch failed: %s",
                            cudaGetErrorString(e));
    return AKASHIC_OK;
}
