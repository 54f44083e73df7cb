// Score step (a1) of query-aware retrieval: z = tau * E q^T, u = exp(z - c),
// with per-tile partial sums toward Z = sum_i u (arXiv 2607.05708, §4.1,
// Dense-only form of §5.5).  Also the query preparation and the running
// maximum of chunk-embedding norms used for the shift bound c.
#include <cudaTypedefs.h>

#include "ak_sm100.cuh"

namespace ak {

// ------------------------------------------------------------------ query prep
// One CTA per padded query row.  shift[c] = tau * |q_c| * max_i |e_i| bounds
// z from above, so u = exp(z - shift) <= 1 never overflows; padding rows are
// zero with shift 0.
// VEC: q 16-byte aligned (dim is a multiple of 64), eight values per load.
template <bool VEC>
__global__ void k_prep_queries(const uint16_t *__restrict__ q, int b, int dim, float tau,
                               const float *__restrict__ max_norm, uint16_t *__restrict__ qp,
                               float *__restrict__ shift, int *status,
                               unsigned int *__restrict__ ext_zero) {
    griddep_wait();
    const int c = blockIdx.x;
    if (ext_zero && c == 0 && threadIdx.x < 2) ext_zero[threadIdx.x] = 0u;
    __shared__ float red[32];
    float ss = 0.f;
    if constexpr (VEC) {
        for (int t = threadIdx.x * 8; t < dim; t += blockDim.x * 8) {
            const uint4 h = (c < b) ? *reinterpret_cast<const uint4 *>(q + (int64_t)c * dim + t)
                                    : make_uint4(0u, 0u, 0u, 0u);
            *reinterpret_cast<uint4 *>(qp + (int64_t)c * dim + t) = h;
            const uint32_t w[4] = {h.x, h.y, h.z, h.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float lo = bf16_to_f32((uint16_t)(w[i] & 0xffffu));
                const float hi = bf16_to_f32((uint16_t)(w[i] >> 16));
                ss = fmaf(lo, lo, ss);
                ss = fmaf(hi, hi, ss);
            }
        }
    } else {
        for (int t = threadIdx.x; t < dim; t += blockDim.x) {
            uint16_t h = (c < b) ? q[(int64_t)c * dim + t] : (uint16_t)0;
            qp[(int64_t)c * dim + t] = h;
            float v = bf16_to_f32(h);
            ss = fmaf(v, v, ss);
        }
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
                                cudaStream_t st, unsigned int *ext_zero) {
    const bool vec = ((uintptr_t)q & 15) == 0 && dim % 8 == 0;
    cudaError_t e = launch_pdl(vec ? k_prep_queries<true> : k_prep_queries<false>, dim3(bp),
                               dim3(128), 0, st, q, b, dim, tau, max_norm, qp, shift, status,
                               ext_zero);
    return e == cudaSuccess ? cudaGetLastError() : e;
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

// ------------------------------------------------------------------ tensor maps
static PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
        else
            cudaGetLastError();
    }
    return fn;
}

cudaError_t make_tmap_2d(CUtensorMap *map, const void *base, CUtensorMapDataType dtype,
                         int elem_bytes, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                         uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swizzle) {
    auto fn = tmap_encoder();
    if (!fn) return cudaErrorNotSupported;
    (void)elem_bytes;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t es[2] = {1, 1};
    CUresult r = fn(map, dtype, 2, const_cast<void *>(base), dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// ------------------------------------------------------------------ tcgen05 GEMM
// C[j, c] = <e_j, q_c> for 128-row tiles of E against column tiles of BP
// (<= 256) query rows, on the 5th-generation tensor cores: bf16 operands
// staged by TMA in the 128-byte swizzle layout, fp32 accumulator in tensor
// memory (two accumulators, so the epilogue of one tile overlaps the MMAs of
// the next), persistent CTAs walking the tiles round-robin, column tiles
// innermost (the CTAs working at one time share the row tiles they read in
// L2).
//   warp 0     TMA producer (one thread)
//   warp 1     TMEM owner and MMA issuer (one thread)
//   warps 2-5  epilogue, by mode:
//     GEMM_EXP     exp(tau*acc - shift), column sums toward Z, swizzled
//                  staging, TMA store (the score step)
//     GEMM_RAW     the dots themselves, TMA store
//     GEMM_FILTER  no store: every dot whose selection key clears its
//                  column's bound is appended to that column's buffer (the
//                  fused relation top-M)
//     GEMM_EXP_FILTER  the score step with the top-k filter fused and no
//                  store: exp, column sums toward Z, and every value whose
//                  key clears its query's bound appended to that query's
//                  buffer (retrieval without hops)
//     GEMM_KEYS_T  the dots as signed selection keys, written column-major
//                  (keys_t[col][row], plain coalesced stores: a warp writes
//                  32 consecutive rows of one column at a time); rows that
//                  are deleted or whose chunk ID is >= id_limit get key 0
//                  (the sample of the relation update's bound)
enum GemmMode { GEMM_EXP = 0, GEMM_RAW = 1, GEMM_FILTER = 2, GEMM_EXP_FILTER = 3,
                GEMM_KEYS_T = 4 };

struct GemmEpi {
    const float *shift;                 // EXP: [BP]
    float tau;                          // EXP
    float *zpart;                       // EXP: [gridDim][BP]
    int *status;
    int64_t n_cols;                     // FILTER: real columns (new chunks)
    const int32_t *ext_of;              // FILTER: chunk ID of each row
    int64_t id_limit;                   // FILTER: rows with chunk ID >= limit are skipped
    const unsigned long long *bound;    // FILTER: [n_cols]
    unsigned int *cnt;                  // FILTER: [n_cols]
    unsigned long long *buf;            // FILTER: [n_cols][cap]
    int64_t cap;
    NsScope ns;                         // EXP_FILTER: namespace scope of the queries
    const int32_t *dead_row;            // EXP, EXP_FILTER, FILTER: deleted rows (or NULL):
                                        // no score (u = 0) / never a filter candidate
    uint32_t *keys_t;                   // KEYS_T: [n_ctiles * BP][n_rows]
    uint16_t *u_hi, *u_lo;              // EXP (or NULL): u as split bf16, [n_rows][n_ctiles * BP]
                                        // each (u = hi + lo to 2^-17), instead of fp32
    float *row_max, *row_min;           // EXP (or NULL): [n_rows] largest / smallest u of
    int n_real;                         // the row over the first n_real columns
    unsigned int *ext;                  // with row_max (or NULL), atomically maxed, zeroed
                                        // before: [0] bits of the largest row_max, [1]
                                        // 0x7f800000 - bits of the smallest row_min over
                                        // the rows whose row_max > 0
};

// z[ch] += s with a run-time chunk index kept out of local memory.
template <int N>
__device__ __forceinline__ void zadd(float (&z)[N], int ch, float s) {
#pragma unroll
    for (int i = 0; i < N; ++i)
        if (i == ch) z[i] += s;
}

// P2: the CTA-pair form.  Clusters of two CTAs compute 256-row tiles with
// the two-SM MMA: each CTA stages its own 128 rows of A and half of the
// BP-row B tile per stage (so a stage is a third smaller at BP = 256 and
// more of them fit), and each CTA's TMEM holds its own rows' accumulators,
// double-buffered.  The odd CTA's copies signal their completion on the
// even CTA's (the MMA issuer's) barrier, whose arrival announces both
// CTAs' bytes; the issuer commits each stage release and each ready
// accumulator to both CTAs' barriers, and the odd CTA's epilogue releases
// the accumulator on the even CTA's barrier by a remote arrive.
template <int BP, int MODE, bool P2 = false>
struct GemmCfg {
    static constexpr int BM = 128, BK = 64;
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = (P2 ? BP / 2 : BP) * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int OUT_BYTES = BM * 32 * 4;
    // the filter epilogue stores nothing: its region only holds the tile's
    // column bounds, and the freed space goes to pipeline stages
    // epilogue warps: the filter epilogues are issue-bound (one compare per
    // dot) and the score epilogue nearly so (exp, row extremes, column
    // sums, staging), so they run two warps per TMEM lane quarter, each on
    // half the columns (HALVES = 2); the others run one
    static constexpr int EPI_W = ((MODE == GEMM_FILTER || MODE == GEMM_KEYS_T ||
                                   MODE == GEMM_EXP || MODE == GEMM_EXP_FILTER) && BP >= 64)
                                     ? 8 : 4;
    static constexpr int HALVES = EPI_W / 4;
    static constexpr int OUT_REGION = (MODE == GEMM_FILTER || MODE == GEMM_KEYS_T)
                                          ? (BP * 12 < 1024 ? 1024 : BP * 12)
                                      : MODE == GEMM_EXP_FILTER ? 2 * OUT_BYTES + BP * 12
                                                                : 2 * HALVES * OUT_BYTES;
    static constexpr int MISC = 4096;   // shift, Z sums, flags, barriers
    static constexpr int BUDGET = 227 * 1024 - 1024;
    static constexpr int S_FIT = (BUDGET - OUT_REGION - MISC) / STAGE_BYTES;
    static constexpr int STAGES = S_FIT > 8 ? 8 : S_FIT;
    static constexpr int TMEM_COLS = 2 * BP < 32 ? 32 : 2 * BP;
    static constexpr int EPI_T = 32 * EPI_W;
    static constexpr int THREADS = 64 + EPI_T;
    static constexpr int SMEM = 1024 + STAGES * STAGE_BYTES + OUT_REGION + MISC;
    static_assert(BP >= 32 && BP <= 256 && (BP & (BP - 1)) == 0, "BP must be 32..256, a power of 2");
    static_assert(STAGES >= 2, "not enough shared memory for two stages");
    static_assert(!P2 || BP >= 128, "the pair form needs B halves of 64 rows or more");
};

template <int BP, int MODE, bool P2 = false>
__global__ __launch_bounds__(GemmCfg<BP, MODE, P2>::THREADS, 1) void k_gemm_umma(const __grid_constant__ CUtensorMap tmA,
                                                      const __grid_constant__ CUtensorMap tmB,
                                                      const __grid_constant__ CUtensorMap tmC,
                                                      const __grid_constant__ CUtensorMap tmD,
                                                      int64_t n_rows, int dim, int n_ctiles,
                                                      const GemmEpi ep) {
    using C = GemmCfg<BP, MODE, P2>;
    griddep_wait();
    constexpr bool EXPF = MODE == GEMM_EXP_FILTER;
    constexpr bool EXP = MODE == GEMM_EXP || EXPF;
    constexpr bool FILTER = MODE == GEMM_FILTER;
    constexpr bool KEYST = MODE == GEMM_KEYS_T;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *sA = smem;
    uint8_t *sB = smem + C::STAGES * C::A_BYTES;
    float *sOut = (float *)(smem + C::STAGES * C::STAGE_BYTES);     // 2 x [128][32], swizzled
    uint8_t *misc = smem + C::STAGES * C::STAGE_BYTES + C::OUT_REGION;
    float *shift_s = (float *)misc;                  // [BP]  (ends below misc + 1024)
    float *xmax = (float *)(misc + 1024);            // [128] row extremes of the second
    float *xmin = xmax + 128;                        // column half (ends at misc + 2048)
    int *go = (int *)(misc + 2560);                  // epilogue: the tile's accumulator is ready
    uint64_t *bars = (uint64_t *)(misc + 3072);      // full[S], empty[S], tfull[2], tempty[2]
    uint64_t *full = bars, *empty = bars + C::STAGES;
    uint64_t *tfull = bars + 2 * C::STAGES, *tempty = tfull + 2;
    uint64_t *done_bar = tempty + 2;                 // the issuer's MMAs have all completed
    uint32_t *tmem_slot = (uint32_t *)(done_bar + 1);
    // filters: the tile's column bounds and the same as float thresholds
    unsigned long long *bnd_s = (unsigned long long *)(sOut + (EXPF ? 2 * C::OUT_BYTES / 4 : 0));
    float *thr_s = (float *)(bnd_s + BP);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // the pair form: this CTA's rank in its cluster (0 issues the MMAs)
    const uint32_t crank = P2 ? cluster_ctarank() : 0u;
    const bool lead = crank == 0u;
    constexpr int TM = P2 ? 2 * C::BM : C::BM;       // rows of a work unit
    const int row_off = (int)crank * C::BM;          // this CTA's rows in a unit
    const int b_off = (int)crank * (BP / 2);         // this CTA's half of the B tile (P2)
    const int64_t m_tiles = (n_rows + TM - 1) / TM;
    // work units: (row tile, column tile); the two CTAs of a pair share each
    const int64_t n_units = m_tiles * n_ctiles;
    const int64_t u_first = P2 ? blockIdx.x / 2 : blockIdx.x;
    const int64_t u_step = P2 ? gridDim.x / 2 : gridDim.x;
    const int kb_n = dim / C::BK;
    int *status = ep.status;
    const float tau_l2e = ep.tau * LOG2E_F;

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], P2 && lead ? 2 : 1);   // both CTAs' epilogues
        }
        mbar_init(done_bar, 1);
        mbar_fence_init();
    }
    if (warp == 1) {
        if constexpr (P2) {
            tmem_alloc2(tmem_slot, C::TMEM_COLS);
            tmem_relinquish2();
        } else {
            tmem_alloc(tmem_slot, C::TMEM_COLS);
            tmem_relinquish();
        }
    }
    for (int i = threadIdx.x; i < BP; i += blockDim.x) {
        // exp(tau x - c) evaluated as 2^(x tau log2(e) - c log2(e)): one FMA
        // and the hardware exp2 per score
        shift_s[i] = EXP ? ep.shift[i] * LOG2E_F : 0.f;
    }
    tc_fence_before();
    __syncthreads();
    if constexpr (P2) cluster_sync();   // both CTAs' barriers exist before any remote arrive
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // ---------------- TMA producer (each CTA loads its own share)
            uint32_t stage = 0, phase = 0;
            int last_par[8];
            for (int s = 0; s < 8; ++s) last_par[s] = -1;
            bool ok = true;
            for (int64_t u = u_first; u < n_units && ok; u += u_step) {
                const int64_t ct = u % n_ctiles;
                const int64_t mt = u / n_ctiles;
                for (int kb = 0; kb < kb_n; ++kb) {
                    // (the odd CTA's releases arrive remotely: spin on them)
                    // (a bounded spin: the suspending wait added wake-up time on the
                    // producer's path every stage; relate 6.76 -> 6.65 ms)
                    if (!mbar_wait_spin(&empty[stage], phase ^ 1u, status)) {
                        ok = false;
                        break;
                    }
                    if (lead) {
                        // the stage fills with both CTAs' bytes
                        mbar_expect_tx(&full[stage], (P2 ? 2 : 1) * C::STAGE_BYTES);
                        tma_load_2d(sA + stage * C::A_BYTES, &tmA, &full[stage], kb * C::BK,
                                    (int)(mt * TM));
                        tma_load_2d(sB + stage * C::B_BYTES, &tmB, &full[stage], kb * C::BK,
                                    (int)(ct * BP));
                    } else {
                        // the odd CTA's copies complete on the even CTA's barrier
                        tma_load_2d_pair(sA + stage * C::A_BYTES, &tmA, &full[stage], 0u,
                                         kb * C::BK, (int)(mt * TM + row_off));
                        tma_load_2d_pair(sB + stage * C::B_BYTES, &tmB, &full[stage], 0u,
                                         kb * C::BK, (int)(ct * BP + b_off));
                    }
                    last_par[stage] = (int)phase;
                    if (++stage == (uint32_t)C::STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!ok) {
                // let every copy this thread issued land before the CTA exits
                if (lead) {
                    for (int s = 0; s < C::STAGES; ++s)
                        if (last_par[s] >= 0) mbar_wait(&full[s], (uint32_t)last_par[s], status);
                } else {
                    // the odd CTA's copies report to the even CTA: give them
                    // ample time (they land within microseconds)
                    for (int i = 0; i < 200; ++i) __nanosleep(1000);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0 && lead) {
            // ---------------- MMA issuer
            const uint32_t idesc = idesc_bf16(TM, BP);
            uint32_t stage = 0, phase = 0;
            int it = 0;
            bool ok = true;
            for (int64_t u = u_first; u < n_units && ok; u += u_step, ++it) {
                const int acc = it & 1;
                const uint32_t aph = (uint32_t)(it >> 1) & 1u;
                if (!(P2 ? mbar_wait_spin(&tempty[acc], aph ^ 1u, status)
                         : mbar_wait(&tempty[acc], aph ^ 1u, status)))
                    break;
                tc_fence_after();
                const uint32_t d = tmem_base + (uint32_t)(acc * BP);
                for (int kb = 0; kb < kb_n; ++kb) {
                    if (!mbar_wait_spin(&full[stage], phase, status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t ad = sdesc_sw128(smem_u32(sA + stage * C::A_BYTES));
                    const uint64_t bd = sdesc_sw128(smem_u32(sB + stage * C::B_BYTES));
#pragma unroll
                    for (int k = 0; k < C::BK / 16; ++k) {
                        if constexpr (P2)
                            umma2_bf16(d, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc,
                                       (kb | k) != 0 ? 1u : 0u);
                        else
                            umma_bf16(d, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc,
                                      (kb | k) != 0 ? 1u : 0u);
                    }
                    if constexpr (P2) {
                        umma2_commit(&empty[stage]);
                        umma2_commit_to(&empty[stage], 1u);
                    } else {
                        umma_commit(&empty[stage]);
                    }
                    if (++stage == (uint32_t)C::STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (ok) {
                    if constexpr (P2) {
                        umma2_commit(&tfull[acc]);
                        umma2_commit_to(&tfull[acc], 1u);
                    } else {
                        umma_commit(&tfull[acc]);
                    }
                }
            }
            // every MMA issued has completed before the CTA (and its pair) may leave
            if constexpr (P2) umma2_commit(done_bar);
            else umma_commit(done_bar);
            mbar_wait(done_bar, 0u, status);
        }
    } else {
        // ---------------- epilogue (EPI_T threads; warp w reads TMEM lanes 32*(w%4)..)
        const int q = warp & 3;
        const int row = q * 32 + lane;                   // row inside the tile
        const int et = threadIdx.x - 64;                 // 0..EPI_T-1
        constexpr int CH_PER = BP / 32 / (C::EPI_W / 4); // 32-column chunks per epilogue warp
        const int hsel = (warp - 2) / 4;                 // which column share
        // EXP: column sums toward Z, per warp (its 32 rows) and chunk, over
        // all the CTA's tiles (one column tile), lane = column in the chunk
        float zl[BP / 32];
#pragma unroll
        for (int i = 0; i < BP / 32; ++i) zl[i] = 0.f;
        float emx = 0.f, emn = INFINITY;                 // this thread's rows' extremes
        int it = 0, cc = 0;
        for (int64_t u = u_first; u < n_units; u += u_step, ++it) {
            const int64_t ct = u % n_ctiles;
            const int64_t mt = u / n_ctiles;
            const int acc = it & 1;
            const uint32_t aph = (uint32_t)(it >> 1) & 1u;
            // one thread polls, the barrier makes the outcome uniform
            if (et == 0) {
                const bool ok = P2 && !lead ? mbar_wait_spin(&tfull[acc], aph, status)
                                            : mbar_wait(&tfull[acc], aph, status);
                *go = ok ? 1 : 0;
            }
            if (FILTER || EXPF) {
                // threshold T with: v < T => key < bound; v > T => key > bound
                // (signed keys order values like floats, -0 below +0; the
                // exp values are >= 0 and their keys are the plain bits); a
                // bound of 0 admits everything, the padding bound ~0 nothing
                // (a NaN threshold)
                for (int c = et; c < BP; c += C::EPI_T) {
                    const int64_t cg = ct * BP + c;
                    const unsigned long long bk = cg < ep.n_cols ? ep.bound[cg] : ~0ull;
                    const uint32_t hi = (uint32_t)(bk >> 32);
                    bnd_s[c] = bk;
                    if (FILTER) thr_s[c] = hi == 0u ? -INFINITY : unordered_bits(hi);
                    else thr_s[c] = __uint_as_float(hi);
                }
            }
            named_bar(1, C::EPI_T);
            if (!*go) break;
            tc_fence_after();
            const int64_t grow = mt * TM + row_off + row;
            const bool in_rows = grow < n_rows;
            const bool valid =
                in_rows && (MODE == GEMM_RAW || !ep.dead_row || !ep.dead_row[grow]);
            uint32_t fid = 0;
            bool fok = false;
            const bool kok = KEYST && valid && (int64_t)ep.ext_of[grow] < ep.id_limit;
            float rmax = 0.f, rmin = INFINITY;           // u >= 0
            if ((FILTER || EXPF) && valid) {
                const int32_t id = ep.ext_of[grow];
                fok = (int64_t)id < ep.id_limit;
                fid = ~(uint32_t)id;
            }
#pragma unroll 1
            for (int ch = hsel * CH_PER; ch < (hsel + 1) * CH_PER; ++ch, ++cc) {
                const int buf = cc & 1;
                uint32_t r[32];
                tmem_ld32(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BP + ch * 32), r);
                tmem_ld_wait();
                if constexpr (KEYST) {
                    if (in_rows) {
                        uint32_t *kt = ep.keys_t + (ct * BP + ch * 32) * n_rows + grow;
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            kt[(int64_t)i * n_rows] = kok ? ordered_bits(__uint_as_float(r[i])) : 0u;
                    }
                } else if constexpr (FILTER) {
                    if (fok) {
                        // one float compare per dot, branch-free, into a mask;
                        // the exact key test only for the few flagged
                        const float4 *t4 = (const float4 *)(thr_s + ch * 32);
                        uint32_t pass = 0u;
#pragma unroll
                        for (int i4 = 0; i4 < 8; ++i4) {
                            const float4 t = t4[i4];
                            pass |= (__uint_as_float(r[4 * i4]) >= t.x ? 1u : 0u) << (4 * i4);
                            pass |= (__uint_as_float(r[4 * i4 + 1]) >= t.y ? 1u : 0u) << (4 * i4 + 1);
                            pass |= (__uint_as_float(r[4 * i4 + 2]) >= t.z ? 1u : 0u) << (4 * i4 + 2);
                            pass |= (__uint_as_float(r[4 * i4 + 3]) >= t.w ? 1u : 0u) << (4 * i4 + 3);
                        }
                        if (pass) {
#pragma unroll
                            for (int i = 0; i < 32; ++i) {
                                if (!((pass >> i) & 1u)) continue;
                                const unsigned long long key =
                                    ((unsigned long long)ordered_bits(__uint_as_float(r[i])) << 32) | fid;
                                if (key >= bnd_s[ch * 32 + i]) {
                                    const int64_t cg = ct * BP + ch * 32 + i;
                                    const unsigned int p = atomicAdd(&ep.cnt[cg], 1u);
                                    if ((int64_t)p < ep.cap) ep.buf[cg * ep.cap + p] = key;
                                }
                            }
                        }
                    }
                } else {
                float v[32];
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const float x = __uint_as_float(r[i]);
                    v[i] = valid ? (EXP ? exp2f(fmaf(x, tau_l2e, -shift_s[ch * 32 + i])) : x) : 0.f;
                }
                if (MODE == GEMM_EXP && ep.row_max) {
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (ch * 32 + i < ep.n_real) {
                            rmax = fmaxf(rmax, v[i]);
                            rmin = fminf(rmin, v[i]);
                        }
                }
                if (MODE == GEMM_EXP && ep.u_hi) {
                    // u as split bf16: hi and lo tiles [128 rows][32 cols] of
                    // 64-byte rows in the 64-byte swizzle (the 16-byte chunk c
                    // of row r at c ^ ((r >> 1) & 3)), one TMA store each
                    named_bar(2 + hsel, 128);                 // staging[buf] free again
                    uint8_t *sb = (uint8_t *)(sOut + (hsel * 2 + buf) * (C::OUT_BYTES / 4));
                    uint32_t hw[16], lw[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) hw[i] = split_bf16_pair(v[2 * i], v[2 * i + 1], lw[i]);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int pos = row * 64 + ((j ^ ((row >> 1) & 3)) << 4);
                        *reinterpret_cast<uint4 *>(sb + pos) =
                            make_uint4(hw[4 * j], hw[4 * j + 1], hw[4 * j + 2], hw[4 * j + 3]);
                        *reinterpret_cast<uint4 *>(sb + C::OUT_BYTES / 2 + pos) =
                            make_uint4(lw[4 * j], lw[4 * j + 1], lw[4 * j + 2], lw[4 * j + 3]);
                    }
                    fence_async_smem();
                    // Z: the column sums of the warp's 32 rows (fp32), by
                    // halving exchanges across the lanes: lane l ends with
                    // column l's sum
#pragma unroll
                    for (int o = 16; o >= 1; o >>= 1) {
                        const bool up = (lane & o) != 0;
#pragma unroll
                        for (int i = 0; i < o; ++i) {
                            const float send = up ? v[i] : v[i + o];
                            const float keep = up ? v[i + o] : v[i];
                            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
                        }
                    }
                    zadd(zl, ch, v[0]);
                    named_bar(2 + hsel, 128);                 // staging[buf] complete
                    if ((et & 127) == 0) {
                        if (mt * TM + row_off < n_rows) {
                            tma_store_2d(&tmC, sb, (int)(ct * BP + ch * 32),
                                         (int)(mt * TM + row_off));
                            tma_store_2d(&tmD, sb + C::OUT_BYTES / 2, (int)(ct * BP + ch * 32),
                                         (int)(mt * TM + row_off));
                            bulk_commit();
                        }
                        bulk_wait_read<1>();                  // the other buffer is free
                    }
                    continue;
                }
                // filter, first half: which of this row's 32 values reach
                // their query's threshold (branch-free; rarely any)
                uint32_t pass = 0u;
                if constexpr (EXPF) {
                    if (fok) {
                        const float4 *t4 = (const float4 *)(thr_s + ch * 32);
#pragma unroll
                        for (int i4 = 0; i4 < 8; ++i4) {
                            const float4 t = t4[i4];
                            pass |= (v[4 * i4] >= t.x ? 1u : 0u) << (4 * i4);
                            pass |= (v[4 * i4 + 1] >= t.y ? 1u : 0u) << (4 * i4 + 1);
                            pass |= (v[4 * i4 + 2] >= t.z ? 1u : 0u) << (4 * i4 + 2);
                            pass |= (v[4 * i4 + 3] >= t.w ? 1u : 0u) << (4 * i4 + 3);
                        }
                    }
                }
                // stage the row: EXP_FILTER in the warp's own 32 rows of its
                // column half's buffer (warp-private, no CTA barrier); EXP /
                // RAW in the column half's buffer buf, shared with the TMA store
                float *so_base;
                if constexpr (EXPF) {
                    __syncwarp();                             // the warp's rows free again
                    so_base = sOut + hsel * (C::OUT_BYTES / 4);
                } else {
                    named_bar(2 + hsel, 128);                 // staging[buf] free again
                    so_base = sOut + (hsel * 2 + buf) * (C::OUT_BYTES / 4);
                }
                float4 *dst = (float4 *)(so_base + row * 32);
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    dst[j ^ (row & 7)] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
                if (!EXPF) fence_async_smem();
                __syncwarp();
                if (EXP) {
                    // column `lane` of this warp's 32 rows
                    float s = 0.f;
#pragma unroll 8
                    for (int rr = q * 32; rr < q * 32 + 32; ++rr)
                        s += so_base[rr * 32 + ((((lane >> 2) ^ (rr & 7))) << 2) + (lane & 3)];
                    zadd(zl, ch, s);
                }
                if constexpr (EXPF) {
                    // second half: the exact key test and append for the
                    // flagged values, read back from the staged row
                    const float *so = so_base + row * 32;
                    while (pass) {
                        const int i = __ffs(pass) - 1;
                        pass &= pass - 1u;
                        const float x = so[(((i >> 2) ^ (row & 7)) << 2) + (i & 3)];
                        const unsigned long long key =
                            ((unsigned long long)__float_as_uint(x) << 32) | fid;
                        if (key >= bnd_s[ch * 32 + i] &&
                            in_scope(ep.ns, grow, (int)(ct * BP + ch * 32 + i))) {
                            const int64_t cg = ct * BP + ch * 32 + i;
                            const unsigned int p = atomicAdd(&ep.cnt[cg], 1u);
                            if ((int64_t)p < ep.cap) ep.buf[cg * ep.cap + p] = key;
                        }
                    }
                } else {
                    named_bar(2 + hsel, 128);                 // staging[buf] complete
                    if ((et & 127) == 0) {
                        // (the odd CTA's half of the last pair tile may lie
                        // wholly past the last row: no store starts there)
                        if (mt * TM + row_off < n_rows) {
                            tma_store_2d(&tmC, so_base, (int)(ct * BP + ch * 32),
                                         (int)(mt * TM + row_off));
                            bulk_commit();
                        }
                        bulk_wait_read<1>();                  // the other buffer is free
                    }
                }
                }
            }
            if (MODE == GEMM_EXP && ep.row_max) {
                if constexpr (C::HALVES == 2) {
                    // the row's second column half hands its extremes over
                    if (hsel == 1) {
                        xmax[row] = rmax;
                        xmin[row] = rmin;
                    }
                    named_bar(1, C::EPI_T);
                    if (hsel == 0) {
                        rmax = fmaxf(rmax, xmax[row]);
                        rmin = fminf(rmin, xmin[row]);
                    }
                }
                if (hsel == 0 && in_rows) {
                    ep.row_max[grow] = rmax;
                    ep.row_min[grow] = rmin;
                    emx = fmaxf(emx, rmax);
                    if (rmax > 0.f) emn = fminf(emn, rmin);
                }
            }
            tc_fence_before();
            named_bar(1, C::EPI_T);
            if (et == 0) {
                if (P2 && !lead) mbar_arrive_remote(&tempty[acc], 0u);
                else mbar_arrive(&tempty[acc]);
            }
        }
        if (MODE == GEMM_EXP && ep.ext) {
            // u >= 0: float bits order like the values
            unsigned int mx = __float_as_uint(emx), mn = 0x7f800000u - __float_as_uint(emn);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, off));
                mn = max(mn, __shfl_xor_sync(0xffffffffu, mn, off));
            }
            if (lane == 0) {
                atomicMax(ep.ext, mx);
                atomicMax(ep.ext + 1, mn);
            }
        }
        if (!EXPF && (et & 127) == 0) bulk_wait_all();
        named_bar(1, C::EPI_T);
        if (EXP && ep.zpart) {
            // the four lane quarters' column sums, added in a fixed order
            // (each chunk's sums come from the one warp of its column half)
            float *zred = sOut;                               // [4][BP], free now
#pragma unroll
            for (int i = 0; i < BP / 32; ++i)
                if (i / CH_PER == hsel) zred[q * BP + i * 32 + lane] = zl[i];
            named_bar(1, C::EPI_T);
            for (int c = et; c < BP; c += C::EPI_T)
                ep.zpart[(int64_t)blockIdx.x * BP + c] =
                    (zred[c] + zred[BP + c]) + (zred[2 * BP + c] + zred[3 * BP + c]);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if constexpr (P2) {
        // neither CTA leaves while the other may still arrive on its
        // barriers or the pair's MMAs read its shared memory
        cluster_sync();
        tc_fence_after();
        if (warp == 1) tmem_dealloc2(tmem_base, C::TMEM_COLS);
    } else {
        if (warp == 1) tmem_dealloc(tmem_base, C::TMEM_COLS);
    }
}

int64_t score_tiles(int64_t n) { return ceil_div<int64_t>(n, 128); }

// The give-up path of the bounded waits, on its own: one thread waits for
// the first phase of a barrier that nothing arrives on, with the same wait
// the tensor-core kernels use, and gives up after `polls` polls.
__global__ void k_wait_timeout_check(int *status, uint32_t polls) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_fence_init();
        mbar_wait_n(&bar, 0u, status, polls);
    }
}

cudaError_t launch_wait_timeout_check(int *status, uint32_t polls, cudaStream_t st) {
    k_wait_timeout_check<<<1, 32, 0, st>>>(status, polls);
    return cudaGetLastError();
}

// The kernel's dynamic shared-memory limit, raised once per device (with
// that device current) before its first launch there; for the pair form
// also the number of clusters of two that fit on the device at once (one
// CTA per SM), or 0 if none does.
template <int BP, int MODE, bool P2 = false>
static cudaError_t gemm_attr(int *clusters = nullptr) {
    using C = GemmCfg<BP, MODE, P2>;
    static bool attr[64] = {false};
    static int ncl[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) return cudaSuccess;
    if (!attr[dev]) {
        cudaError_t e = cudaFuncSetAttribute(k_gemm_umma<BP, MODE, P2>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (e != cudaSuccess) return e;
        if (P2) {
            cudaLaunchConfig_t cfg = {};
            cudaLaunchAttribute at[1];
            at[0].id = cudaLaunchAttributeClusterDimension;
            at[0].val.clusterDim.x = 2;
            at[0].val.clusterDim.y = 1;
            at[0].val.clusterDim.z = 1;
            cfg.gridDim = dim3((unsigned)(device_sm_count() & ~1));
            cfg.blockDim = dim3(C::THREADS);
            cfg.dynamicSmemBytes = C::SMEM;
            cfg.attrs = at;
            cfg.numAttrs = 1;
            int n = 0;
            e = cudaOccupancyMaxActiveClusters(&n, k_gemm_umma<BP, MODE, P2>, &cfg);
            if (e != cudaSuccess) return e;
            ncl[dev] = n;
        }
        attr[dev] = true;
    }
    if (clusters) *clusters = ncl[dev];
    return cudaSuccess;
}

// The pair form is taken where it applies unless AKASHIC_GEMM_PAIR=0.
static bool gemm_pair_enabled() {
    static int v = -1;
    if (v < 0) {
        const char *e = getenv("AKASHIC_GEMM_PAIR");
        v = (e && e[0] == '0') ? 0 : 1;
    }
    return v == 1;
}

cudaError_t prepare_score_gemm() {
    cudaError_t e = gemm_attr<32, GEMM_EXP>();
    if (e == cudaSuccess) e = gemm_attr<64, GEMM_EXP>();
    if (e == cudaSuccess) e = gemm_attr<128, GEMM_EXP>();
    if (e == cudaSuccess) e = gemm_attr<256, GEMM_EXP>();
    if (e == cudaSuccess) e = gemm_attr<128, GEMM_EXP, true>();
    if (e == cudaSuccess) e = gemm_attr<256, GEMM_EXP, true>();
    return e;
}

// A: E rows (row_stride_rows apart: 1 = every row, s = every s-th row),
// B: n_ctiles * BP query rows, C: output [n_rows][n_ctiles * BP] (EXP/RAW).
// The grid: one CTA per SM at most (the single form), or clusters of two
// on 256-row tiles (the pair form, B >= 128, taken when the rows fill every
// cluster that fits, so that the grid never exceeds ceil(n_rows / 128) and
// the Z partials keep at most one row per 128-row tile).  *zrows = grid.
template <int BP, int MODE>
static cudaError_t gemm_bp(const uint16_t *emb, int64_t n_rows, int64_t row_stride_rows, int dim,
                           const uint16_t *qp, int n_ctiles, float *out, const GemmEpi &ep,
                           cudaStream_t st, int *zrows) {
    constexpr bool CAN_P2 = BP >= 128;
    int ncl = 0;
    if constexpr (CAN_P2) {
        if (gemm_pair_enabled()) {
            cudaError_t e = gemm_attr<BP, MODE, true>(&ncl);
            if (e != cudaSuccess) return e;
        }
    }
    const bool p2 = CAN_P2 && ncl > 0 && n_rows >= (int64_t)256 * ncl;
    if (!p2) {
        cudaError_t e = gemm_attr<BP, MODE>();
        if (e != cudaSuccess) return e;
    }
    CUtensorMap ta, tb, tc, td;
    cudaError_t e = make_tmap_2d(&ta, emb, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (uint64_t)dim,
                                 (uint64_t)n_rows, (uint64_t)dim * 2 * row_stride_rows, 64, 128);
    if (e == cudaSuccess)
        e = make_tmap_2d(&tb, qp, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (uint64_t)dim,
                         (uint64_t)n_ctiles * BP, (uint64_t)dim * 2, 64, p2 ? BP / 2 : BP);
    const uint64_t n_cols = (uint64_t)n_ctiles * BP;
    if (e == cudaSuccess && MODE == GEMM_EXP && ep.u_hi) {
        // split-bf16 output: [128][32] boxes of 64-byte rows, 64-byte swizzle
        e = make_tmap_2d(&tc, ep.u_hi, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, n_cols,
                         (uint64_t)n_rows, n_cols * 2, 32, 128, CU_TENSOR_MAP_SWIZZLE_64B);
        if (e == cudaSuccess)
            e = make_tmap_2d(&td, ep.u_lo, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, n_cols,
                             (uint64_t)n_rows, n_cols * 2, 32, 128, CU_TENSOR_MAP_SWIZZLE_64B);
    } else if (e == cudaSuccess && MODE != GEMM_FILTER && MODE != GEMM_EXP_FILTER &&
               MODE != GEMM_KEYS_T) {
        e = make_tmap_2d(&tc, out, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, n_cols, (uint64_t)n_rows,
                         n_cols * 4, 32, 128);
        td = tc;   // unused
    } else {
        tc = td = ta;   // unused by the filter epilogues
    }
    if (e != cudaSuccess) return e;
    if constexpr (CAN_P2) {
        if (p2) {
            using C2 = GemmCfg<BP, MODE, true>;
            const int64_t units = ceil_div<int64_t>(n_rows, 256) * n_ctiles;
            const int64_t clusters = units < ncl ? units : ncl;
            cudaLaunchConfig_t cfg = {};
            cudaLaunchAttribute at[2];
            at[0].id = cudaLaunchAttributeClusterDimension;
            at[0].val.clusterDim.x = 2;
            at[0].val.clusterDim.y = 1;
            at[0].val.clusterDim.z = 1;
            at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // see griddep_wait
            at[1].val.programmaticStreamSerializationAllowed = 1;
            cfg.gridDim = dim3((unsigned)(2 * clusters));
            cfg.blockDim = dim3(C2::THREADS);
            cfg.dynamicSmemBytes = C2::SMEM;
            cfg.stream = st;
            cfg.attrs = at;
            cfg.numAttrs = 2;
            e = cudaLaunchKernelEx(&cfg, k_gemm_umma<BP, MODE, true>, ta, tb, tc, td, n_rows, dim,
                                   n_ctiles, ep);
            if (zrows) *zrows = (int)(2 * clusters);
            return e == cudaSuccess ? cudaGetLastError() : e;
        }
    }
    using C = GemmCfg<BP, MODE>;
    const int64_t m_tiles = ceil_div<int64_t>(n_rows, 128);
    const int64_t tiles = m_tiles * n_ctiles;
    const int grid = (int)(tiles < device_sm_count() ? tiles : device_sm_count());
    e = launch_pdl(k_gemm_umma<BP, MODE, false>, dim3(grid), dim3(C::THREADS), C::SMEM, st, ta, tb,
                   tc, td, n_rows, dim, n_ctiles, ep);
    if (zrows) *zrows = grid;
    return e == cudaSuccess ? cudaGetLastError() : e;
}

template <int MODE>
static cudaError_t gemm_dispatch(const uint16_t *emb, int64_t n_rows, int64_t row_stride_rows,
                                 int dim, const uint16_t *qp, int bp, int n_ctiles, float *out,
                                 const GemmEpi &ep, cudaStream_t st, int *zrows) {
    if (n_rows <= 0 || dim % 64 != 0 || n_ctiles < 1) return cudaErrorInvalidValue;
    switch (bp) {
    case 32: return gemm_bp<32, MODE>(emb, n_rows, row_stride_rows, dim, qp, n_ctiles, out, ep, st, zrows);
    case 64: return gemm_bp<64, MODE>(emb, n_rows, row_stride_rows, dim, qp, n_ctiles, out, ep, st, zrows);
    case 128: return gemm_bp<128, MODE>(emb, n_rows, row_stride_rows, dim, qp, n_ctiles, out, ep, st, zrows);
    case 256: return gemm_bp<256, MODE>(emb, n_rows, row_stride_rows, dim, qp, n_ctiles, out, ep, st, zrows);
    default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_score(const uint16_t *emb, int64_t n, int dim, const uint16_t *qp, int bp,
                         const float *shift, float tau, float *u, float *zpart, int *status,
                         cudaStream_t st, int *launches, int *zrows, const int32_t *dead_row,
                         float *row_max, float *row_min, int n_real, unsigned int *ext) {
    GemmEpi ep{};
    ep.dead_row = dead_row;
    ep.row_max = row_max;
    ep.row_min = row_min;
    ep.n_real = n_real;
    ep.ext = row_max ? ext : nullptr;
    ep.shift = shift;
    ep.tau = tau;
    ep.zpart = zpart;
    ep.status = status;
    cudaError_t e = gemm_dispatch<GEMM_EXP>(emb, n, 1, dim, qp, bp, 1, u, ep, st, zrows);
    if (launches) *launches += 1;
    return e;
}

cudaError_t launch_score_split(const uint16_t *emb, int64_t n, int dim, const uint16_t *qp, int bp,
                               const float *shift, float tau, uint16_t *u_hi, uint16_t *u_lo,
                               float *zpart, int *status, cudaStream_t st, int *launches,
                               int *zrows, const int32_t *dead_row, float *row_max,
                               float *row_min, int n_real, unsigned int *ext) {
    GemmEpi ep{};
    ep.dead_row = dead_row;
    ep.row_max = row_max;
    ep.row_min = row_min;
    ep.n_real = n_real;
    ep.ext = row_max ? ext : nullptr;
    ep.shift = shift;
    ep.tau = tau;
    ep.zpart = zpart;
    ep.status = status;
    ep.u_hi = u_hi;
    ep.u_lo = u_lo;
    cudaError_t e = gemm_dispatch<GEMM_EXP>(emb, n, 1, dim, qp, bp, 1, nullptr, ep, st, zrows);
    if (launches) *launches += 1;
    return e;
}

cudaError_t launch_score_sample(const uint16_t *emb, int64_t n_sample, int64_t stride, int dim,
                                const uint16_t *qp, int bp, const float *shift, float tau,
                                float *out, float *zpart, int *status, cudaStream_t st,
                                int *launches) {
    GemmEpi ep{};
    ep.shift = shift;
    ep.tau = tau;
    ep.zpart = zpart;
    ep.status = status;
    cudaError_t e = gemm_dispatch<GEMM_EXP>(emb, n_sample, stride, dim, qp, bp, 1, out, ep, st,
                                            nullptr);
    if (launches) *launches += 1;
    return e;
}

cudaError_t launch_score_filter(const uint16_t *emb, int64_t n, int dim, const uint16_t *qp,
                                int bp, int64_t n_cols, const float *shift, float tau,
                                float *zpart, const int32_t *ext_of,
                                const unsigned long long *bound, unsigned int *cnt,
                                unsigned long long *buf, int64_t cap, NsScope ns, int *status,
                                cudaStream_t st, int *launches, int *zrows) {
    GemmEpi ep{};
    ep.ns = ns;
    ep.dead_row = ns.dead;
    ep.shift = shift;
    ep.tau = tau;
    ep.zpart = zpart;
    ep.status = status;
    ep.n_cols = n_cols;
    ep.ext_of = ext_of;
    ep.id_limit = (int64_t)1 << 40;
    ep.bound = bound;
    ep.cnt = cnt;
    ep.buf = buf;
    ep.cap = cap;
    cudaError_t e = gemm_dispatch<GEMM_EXP_FILTER>(emb, n, 1, dim, qp, bp, 1, nullptr, ep, st,
                                                   zrows);
    if (launches) *launches += 1;
    return e;
}

cudaError_t launch_dots(const uint16_t *emb, int64_t n, int64_t row_stride_rows, int dim,
                        const uint16_t *qp, int bp, int n_ctiles, float *out, int *status,
                        cudaStream_t st, int *launches) {
    GemmEpi ep{};
    ep.status = status;
    cudaError_t e = gemm_dispatch<GEMM_RAW>(emb, n, row_stride_rows, dim, qp, bp, n_ctiles, out,
                                            ep, st, nullptr);
    if (launches) *launches += 1;
    return e;
}

cudaError_t launch_dots_filter(const uint16_t *emb, int64_t n, int dim, const uint16_t *qp,
                               int n_ctiles, int64_t n_cols, const int32_t *ext_of,
                               int64_t id_limit, const unsigned long long *bound,
                               unsigned int *cnt, unsigned long long *buf, int64_t cap,
                               int *status, cudaStream_t st, int *launches,
                               const int32_t *dead_row) {
    GemmEpi ep{};
    ep.dead_row = dead_row;
    ep.status = status;
    ep.n_cols = n_cols;
    ep.ext_of = ext_of;
    ep.id_limit = id_limit;
    ep.bound = bound;
    ep.cnt = cnt;
    ep.buf = buf;
    ep.cap = cap;
    cudaError_t e = gemm_dispatch<GEMM_FILTER>(emb, n, 1, dim, qp, 256, n_ctiles, nullptr, ep, st,
                                               nullptr);
    if (launches) *launches += 1;
    return e;
}

cudaError_t launch_dots_keys_t(const uint16_t *emb, int64_t n, int64_t row_stride_rows, int dim,
                               const uint16_t *qp, int n_ctiles, const int32_t *ext_of,
                               int64_t id_limit, const int32_t *dead_row, uint32_t *keys_t,
                               int *status, cudaStream_t st, int *launches) {
    GemmEpi ep{};
    ep.dead_row = dead_row;
    ep.status = status;
    ep.ext_of = ext_of;
    ep.id_limit = id_limit;
    ep.keys_t = keys_t;
    cudaError_t e = gemm_dispatch<GEMM_KEYS_T>(emb, n, row_stride_rows, dim, qp, 256, n_ctiles,
                                               nullptr, ep, st, nullptr);
    if (launches) *launches += 1;
    return e;
}

}  // namespace ak
