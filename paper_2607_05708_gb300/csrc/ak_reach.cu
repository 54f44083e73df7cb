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
#include <cuda_bf16.h>

#include "ak_common.cuh"
#include "ak_sm100.cuh"

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
// The plan of a call, on the device: plan[0] = 1 when the candidates
// suffice (no other row reaches the floor, at least k of them do, and at
// least k candidates exist), else 0 and the hops run; plan[1] = nk, the
// flagged count; plan[2 .. 2 + nk) the flagged slots in ascending order;
// plan[REACH_PLAN_WIDE] = 1 when one of them is 64 or above.  Run by one
// CTA of at least REACH_T threads (every thread calls it).
__device__ void reach_build_plan(const int32_t *keep, int bad, int t_cnt, int k, int32_t *plan) {
    __shared__ int pre[REACH_T];
    const int t = threadIdx.x;
    const int f = t < REACH_T && keep[t] != 0 ? 1 : 0;
    if (t < REACH_T) pre[t] = f;
    __syncthreads();
    for (int o = 1; o < REACH_T; o <<= 1) {          // inclusive scan
        const int v = t < REACH_T && t >= o ? pre[t - o] : 0;
        __syncthreads();
        if (t < REACH_T) pre[t] += v;
        __syncthreads();
    }
    if (f) plan[2 + pre[t] - 1] = t;
    if (t == REACH_T - 1) {
        const int nk = pre[t];
        plan[1] = nk;
        plan[0] = (bad == 0 && nk >= k && t_cnt >= k) ? 1 : 0;
        // a flagged slot in the upper half: the candidates' pass loads all
        // 128 coefficient rows, else the first 64
        plan[REACH_PLAN_WIDE] = nk - pre[REACH_T / 2 - 1] > 0 ? 1 : 0;
    }
}

// The floor: the k-th largest lower bound over the n_lb heaviest split
// rows (each query's k-th largest final score reaches it: those k rows
// score at least their lb for every query), computed for those rows only;
// one CTA, one (lb bits, position) key per thread, a descending bitonic
// network (partners within a warp by shuffles, farther ones through a
// ping-pong pair of shared arrays).  Also clears the flags' scratch.
__global__ __launch_bounds__(1024) void k_reach_floor(const ReachFlags f) {
    __shared__ unsigned long long xk[2][1024];
    griddep_wait();
    const int t = threadIdx.x;
    if (t < REACH_T + 2) f.ws[t] = 0;                  // keep[], bad, done
    const float lmin = ext_lmin(f.ext);
    unsigned long long key =
        t < f.n_lb ? ((unsigned long long)__float_as_uint(row_lower_bound(
                          f.l0, f.mdn, f.n, f.H, f.alpha, lmin, f.split_row[f.split_order[t]]))
                      << 32) | (unsigned long long)(uint32_t)t
                   : 0ull;
    int cur = 0;
    for (int size = 2; size <= 1024; size <<= 1)
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
            const bool keep_max = ((t & size) == 0) == ((t & stride) == 0);
            key = keep_max ? (key > other ? key : other) : (key < other ? key : other);
        }
    if (t == f.k - 1)   // keys now descend with the thread index
        *f.floor_out = f.n_lb >= f.k ? __uint_as_float((uint32_t)(key >> 32)) : 0.f;
}

// Rows whose upper bound reaches the floor: a candidate's slot is flagged,
// any other row counted in bad; the last CTA to finish builds the plan.
__global__ __launch_bounds__(256) void k_reach_flags(const ReachFlags f) {
    __shared__ int last;
    griddep_wait();
    int32_t *keep = f.ws, *bad = f.ws + REACH_T, *done = f.ws + REACH_T + 1;
    const float floor_ = *f.floor_out, umax = ext_umax(f.ext);
    int nb = 0;
    auto visit = [&](int64_t j, float ub) {
        if (ub >= floor_) {
            const int32_t t = f.map[j];
            if (t >= 0) keep[t] = 1;
            else ++nb;
        }
    };
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    if ((f.n & 3) == 0) {
        // four rows a thread: 16-byte loads of u's row maxima and of each
        // mass level, the bound evaluated per row as row_upper_bound does
        const int64_t n4 = f.n >> 2;
        for (int64_t q = tid; q < n4; q += stride) {
            float4 c = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int t = f.H; t >= 1; --t) {
                const float4 m =
                    __ldg(reinterpret_cast<const float4 *>(f.mup + (int64_t)t * f.n) + q);
                c.x = f.alpha * (c.x + m.x);
                c.y = f.alpha * (c.y + m.y);
                c.z = f.alpha * (c.z + m.z);
                c.w = f.alpha * (c.w + m.w);
            }
            const float4 u = reinterpret_cast<const float4 *>(f.u0)[q];
            visit(4 * q, fmaf(umax, c.x, u.x) * (1.f + 1e-5f));
            visit(4 * q + 1, fmaf(umax, c.y, u.y) * (1.f + 1e-5f));
            visit(4 * q + 2, fmaf(umax, c.z, u.z) * (1.f + 1e-5f));
            visit(4 * q + 3, fmaf(umax, c.w, u.w) * (1.f + 1e-5f));
        }
    } else {
        for (int64_t j = tid; j < f.n; j += stride)
            visit(j, row_upper_bound(f.u0, f.mup, f.n, f.H, f.alpha, umax, j));
    }
    if (nb) atomicAdd(bad, nb);
    __threadfence();                                   // flags before the count
    __syncthreads();
    if (threadIdx.x == 0) last = atomicAdd(done, 1) == (int)gridDim.x - 1;
    __syncthreads();
    if (!last) return;
    __threadfence();                                   // every CTA's flags are visible
    const volatile int32_t *vk = keep;
    __shared__ int32_t kf[REACH_T];
    if (threadIdx.x < REACH_T) kf[threadIdx.x] = vk[threadIdx.x];
    __syncthreads();
    reach_build_plan(kf, *(volatile int *)bad, *f.t_cnt, f.k, f.plan);
}

cudaError_t launch_reach_flags(const ReachFlags &f, cudaStream_t st, int *launches) {
    if (f.n_lb > 1024 || f.k < 1) return cudaErrorInvalidValue;
    cudaError_t e = launch_pdl(k_reach_floor, dim3(1), dim3(1024), 0, st, f);
    if (e != cudaSuccess) return e;
    // four rows per thread (one where n is not a multiple of 4): a few
    // independent loads per row, so the rows in flight set the rate; a
    // quarter of the CTAs also takes three quarters of the done counter's
    // atomics off the tail
    const int64_t g = ceil_div<int64_t>(f.n, (f.n & 3) == 0 ? 1024 : 256);
    e = launch_pdl(k_reach_flags, dim3((unsigned)(g > 0 ? g : 1)), dim3(256), 0, st, f);
    if (launches) *launches += 2;
    return e == cudaSuccess ? cudaGetLastError() : e;
}

// ------------------------------------------------------------------ tensor-core terms
// partial[cta][i][b] = sum over the CTA's rows k of coef[k][i] u[k][b] for
// every candidate slot i, on tcgen05 with split-bf16 operands:
//   coef = A_hi + A_lo,  u = B_hi + B_lo  (each lo the bf16 rounding of the
//   rest, so hi + lo holds 16 significant bits),
//   coef u ~= A_hi B_hi + A_hi B_lo + A_lo B_hi,
// three MMAs per 16-row slice into an fp32 accumulator in TMEM (the
// dropped A_lo B_lo term is below 2^-16 of the product).
//   A = the combined coefficients sum_t alpha^t C_t, packed by
//       k_reach_pack as [REACH_T slots][n_pad rows] bf16 (hi, lo), loaded
//       by TMA as K-major tiles [128 slots][64 rows] in the 128-byte swizzle;
//   B = u as the score GEMM wrote it, split bf16 [n rows][BP queries] (hi,
//       lo), loaded by TMA as MN-major tiles [64 rows][BP queries]: boxes of
//       64 rows x 64 queries in the 128-byte swizzle (128 bytes a row, the
//       16-byte chunk c of row r at c ^ (r % 8)), i.e. atoms of 8 rows x 64
//       queries, the BP / 64 boxes RM_BK * 128 bytes apart.
// D[slot][query] (M = 128 slots = TMEM lanes, N = BP queries = columns).
// The tensor core's accumulation of many positive terms drifts (each add
// into the fp32 accumulator may round the same way), so an accumulator
// takes only RM_CHUNK stages (1024 rows, 192 MMAs): two accumulators
// alternate, and the flush warps add each finished one into the CTA's
// partial with ordinary round-to-nearest fp32 adds while the MMAs fill the
// other.  The operands' loads carry an L2 evict-first hint and the partial
// rows' loads and stores an evict-last one, so that the partials stay in L2
// while u streams past; slots 64 and above are flushed only when the plan
// is wide.
// Warps: 0 TMA producer (A and B), 1 MMA issuer, 2..9 flush (warp w reads
// TMEM lanes 32 (w % 4) .., column half (w - 2) / 4).  Both operands
// arrive by TMA, so the bytes in flight are the two stages' 192 KB of
// shared memory, not registers.  Each CTA takes a contiguous range of
// 64-row stages.
constexpr int RM_BK = 64;                // store rows (K) per stage
constexpr int RM_M = REACH_T;            // candidate slots (M)
constexpr int RM_STAGES = 2;
constexpr int RM_FLUSH_W = 8;            // flush warps
constexpr int RM_THREADS = 64 + 32 * RM_FLUSH_W;
constexpr int RM_CHUNK = 16;             // stages per accumulator

template <int BP>
struct RmCfg {
    static constexpr int A_BYTES = RM_M * RM_BK * 2;             // one of hi / lo
    static constexpr int B_BYTES = BP * RM_BK * 2;               // one of hi / lo
    static constexpr int STAGE_BYTES = 2 * A_BYTES + 2 * B_BYTES;
    static constexpr uint32_t LBO = RM_BK * 128;                 // between query atoms
    static constexpr uint32_t SBO = 8 * 128;                     // between 8-row groups
    static constexpr int SMEM = 1024 + RM_STAGES * STAGE_BYTES + 256;
    static constexpr int PARTS = RM_FLUSH_W / 4;     // column parts of a flush
    static constexpr int TMEM_COLS = 2 * BP; // two accumulators
    static_assert(BP == 128 || BP == 256, "query widths 128 and 256");
    static_assert(SMEM <= 227 * 1024, "shared memory");
};

template <int BP>
__global__ __launch_bounds__(RM_THREADS, 1) void k_reach_mma(
    const __grid_constant__ CUtensorMap tmAhi, const __grid_constant__ CUtensorMap tmAlo,
    const __grid_constant__ CUtensorMap tmAhi64, const __grid_constant__ CUtensorMap tmAlo64,
    const __grid_constant__ CUtensorMap tmBhi, const __grid_constant__ CUtensorMap tmBlo,
    int64_t n, const int32_t *__restrict__ plan, float *__restrict__ partial, int *status) {
    using C = RmCfg<BP>;
    griddep_wait();
    if (plan[0] == 0) return;                          // the hops run instead
    // every flagged slot below 64: only the first 64 coefficient rows are
    // loaded (rows 64..127 of the A tiles keep whatever they hold, and
    // the accumulator rows they feed are never read)
    const bool wide = plan[REACH_PLAN_WIDE] != 0;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t *full = (uint64_t *)(smem + RM_STAGES * C::STAGE_BYTES);
    uint64_t *empty = full + RM_STAGES;               // the MMAs' commit
    uint64_t *dfull = empty + RM_STAGES;              // [2] accumulator complete
    uint64_t *dfree = dfull + 2;                      // [2] accumulator flushed (RM_FLUSH_W)
    uint32_t *tmem_slot = (uint32_t *)(dfree + 2);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    auto a_hi = [&](int s) { return smem + s * C::STAGE_BYTES; };
    auto a_lo = [&](int s) { return smem + s * C::STAGE_BYTES + C::A_BYTES; };
    auto b_hi = [&](int s) { return smem + s * C::STAGE_BYTES + 2 * C::A_BYTES; };
    auto b_lo = [&](int s) { return smem + s * C::STAGE_BYTES + 2 * C::A_BYTES + C::B_BYTES; };

    const int64_t stages_total = (n + RM_BK - 1) / RM_BK;
    const int64_t per = (stages_total + gridDim.x - 1) / gridDim.x;
    const int64_t s0 = (int64_t)blockIdx.x * per;
    const int64_t s1 = s0 + per < stages_total ? s0 + per : stages_total;
    const int64_t ns = s1 > s0 ? s1 - s0 : 0;
    const int64_t n_chunks = (ns + RM_CHUNK - 1) / RM_CHUNK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < RM_STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&dfull[a], 1);
            mbar_init(&dfree[a], RM_FLUSH_W);
        }
        mbar_fence_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, C::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        if (lane == 0 && ns > 0) {
            // ---------------- TMA producer: A hi / lo [128 slots][64 rows],
            // B hi / lo [64 rows][BP queries] as BP / 64 boxes each
            uint32_t stage = 0, phase = 0;
            int last_par[RM_STAGES];
            for (int s = 0; s < RM_STAGES; ++s) last_par[s] = -1;
            bool ok = true;
            // both operands are read once a call: evict them first, so that
            // they do not push the CTAs' partial rows out of L2
            const uint64_t pol = l2_evict_first_policy();
            for (int64_t t = 0; t < ns; ++t) {
                if (!mbar_wait_spin(&empty[stage], phase ^ 1u, status)) {
                    ok = false;
                    break;
                }
                mbar_expect_tx(&full[stage],
                               (wide ? 2 * C::A_BYTES : C::A_BYTES) + 2 * C::B_BYTES);
                const int kx = (int)((s0 + t) * RM_BK);
                tma_load_2d_hint(a_hi(stage), wide ? &tmAhi : &tmAhi64, &full[stage], kx, 0, pol);
                tma_load_2d_hint(a_lo(stage), wide ? &tmAlo : &tmAlo64, &full[stage], kx, 0, pol);
#pragma unroll
                for (int c = 0; c < BP / 64; ++c) {
                    tma_load_2d_hint(b_hi(stage) + c * C::LBO, &tmBhi, &full[stage], 64 * c, kx,
                                     pol);
                    tma_load_2d_hint(b_lo(stage) + c * C::LBO, &tmBlo, &full[stage], 64 * c, kx,
                                     pol);
                }
                last_par[stage] = (int)phase;
                if (++stage == RM_STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok)   // let every copy this thread issued land before the CTA exits
                for (int s = 0; s < RM_STAGES; ++s)
                    if (last_par[s] >= 0) mbar_wait(&full[s], (uint32_t)last_par[s], status);
        }
    } else if (warp == 1) {
        if (lane == 0 && ns > 0) {
            // ---------------- MMA issuer: three products per 16-row slice
            const uint32_t idesc = idesc_bf16_m128(BP) | IDESC_B_MN_MAJOR;
            uint32_t stage = 0, phase = 0;
            bool ok = true;
            for (int64_t t = 0; t < ns && ok; ++t) {
                const int64_t c = t / RM_CHUNK;
                const int acc = (int)(c & 1);
                const bool first = t % RM_CHUNK == 0;
                const bool last = t % RM_CHUNK == RM_CHUNK - 1 || t == ns - 1;
                // the accumulator is free once the flush warps emptied its
                // previous chunk (c - 2)
                if (first && !mbar_wait(&dfree[acc], (uint32_t)((c >> 1) & 1) ^ 1u, status)) break;
                if (!mbar_wait_spin(&full[stage], phase, status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem_base + (uint32_t)(acc * BP);
                const uint64_t ah = sdesc_sw128(smem_u32(a_hi(stage)));
                const uint64_t al = sdesc_sw128(smem_u32(a_lo(stage)));
                const uint64_t bh = sdesc_mn_sw128(smem_u32(b_hi(stage)), C::LBO, C::SBO);
                const uint64_t bl = sdesc_mn_sw128(smem_u32(b_lo(stage)), C::LBO, C::SBO);
#pragma unroll
                for (int k = 0; k < RM_BK / 16; ++k) {
                    // A: 16 K values = 32 bytes further along the row; B: two
                    // 8-row groups further down
                    const uint64_t ao = (uint64_t)(2 * k), bo = (uint64_t)(2 * C::SBO * k) >> 4;
                    umma_bf16(d, ah + ao, bh + bo, idesc, (first && k == 0) ? 0u : 1u);
                    umma_bf16(d, ah + ao, bl + bo, idesc, 1u);
                    umma_bf16(d, al + ao, bh + bo, idesc, 1u);
                }
                umma_commit(&empty[stage]);
                if (last) umma_commit(&dfull[acc]);
                if (++stage == RM_STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
        }
    } else {
        // ---------------- flush warps: each finished accumulator into the
        // CTA's partial rows (the first chunk stores, the later ones add)
        const int fw = warp - 2;
        const int q = warp & 3;                       // TMEM lanes 32 q ..
        const int part = fw >> 2;                     // column part
        const int slot = q * 32 + lane;
        constexpr int PW = BP / C::PARTS;             // columns of a part
        float *o = partial + ((int64_t)blockIdx.x * REACH_T + slot) * BP + part * PW;
        // slots 64..127 are read only when the plan is wide
        const bool live = wide || q < 2;
        // the partial rows are re-read every chunk: keep them in L2
        const uint64_t pol = l2_evict_last_policy();
        if (ns == 0 && live) {
            for (int b = 0; b < PW; b += 4)
                *reinterpret_cast<float4 *>(o + b) = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        for (int64_t c = 0; c < n_chunks; ++c) {
            const int acc = (int)(c & 1);
            int f_ok = lane == 0 ? (mbar_wait(&dfull[acc], (uint32_t)((c >> 1) & 1), status) ? 1 : 0)
                                 : 0;
            f_ok = __shfl_sync(0xffffffffu, f_ok, 0);
            if (!f_ok) break;
            tc_fence_after();
#pragma unroll 1
            for (int ch = 0; ch < (live ? PW / 32 : 0); ++ch) {
                uint32_t r[32];
                tmem_ld32(tmem_base + ((uint32_t)(q * 32) << 16) +
                              (uint32_t)(acc * BP + part * PW + ch * 32),
                          r);
                tmem_ld_wait();
                float4 *dst = reinterpret_cast<float4 *>(o + ch * 32);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    float4 v = make_float4(__uint_as_float(r[4 * i]), __uint_as_float(r[4 * i + 1]),
                                           __uint_as_float(r[4 * i + 2]),
                                           __uint_as_float(r[4 * i + 3]));
                    if (c > 0) {
                        const float4 p = ld_f4_hint(dst + i, pol);
                        v.x += p.x;
                        v.y += p.y;
                        v.z += p.z;
                        v.w += p.w;
                    }
                    st_f4_hint(dst + i, v, pol);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&dfree[acc]);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem_base, C::TMEM_COLS);
}

// coef_hi / coef_lo [REACH_T][n_pad] bf16: row i = candidate slot i's
// combined coefficient sum_t alpha^t C_t[k][i] (Horner over t) split into
// hi + lo, zero for k >= n.  One CTA per 64 rows k: the rows' slots are
// read contiguously (coalesced), transposed through shared memory and
// written along k (coalesced).
__global__ __launch_bounds__(256) void k_reach_pack(const float *__restrict__ C, int64_t n,
                                                    int64_t n_pad, int H, float alpha,
                                                    uint16_t *__restrict__ hi,
                                                    uint16_t *__restrict__ lo) {
    __shared__ float tile[64][REACH_T + 1];
    const int64_t k0 = (int64_t)blockIdx.x * 64;
    for (int x = threadIdx.x; x < 64 * REACH_T; x += blockDim.x) {
        const int kk = x / REACH_T, i = x % REACH_T;
        const int64_t k = k0 + kk;
        float c = 0.f;
        if (k < n) {
            const int64_t at = k * REACH_T + i;
            for (int t = H; t >= 1; --t) c = alpha * (c + C[(int64_t)(t - 1) * n * REACH_T + at]);
        }
        tile[kk][i] = c;
    }
    __syncthreads();
    for (int x = threadIdx.x; x < 32 * REACH_T; x += blockDim.x) {
        const int i = x / 32, kk = 2 * (x % 32);
        const int64_t k = k0 + kk;
        uint32_t l;
        const uint32_t h = split_bf16_pair(tile[kk][i], tile[kk + 1][i], l);
        *reinterpret_cast<uint32_t *>(hi + (int64_t)i * n_pad + k) = h;
        *reinterpret_cast<uint32_t *>(lo + (int64_t)i * n_pad + k) = l;
    }
}


// Final score of each flagged candidate for each real query column: its u
// plus the CTAs' partials, appended as a filter key (score bits, ~chunk ID)
// to the column's buffer; the buffer then holds exactly them.  bp / 64
// blocks per candidate slot of the plan, each on 64 query columns (blocks
// past nk, and every block when the plan says the hops run, return at
// once): thread t takes column t % 64 of its block's and every 16th
// partial from t / 64 on (coalesced rows of the partials), and the groups
// are added in group order (the same order on every run).
constexpr int EMIT_Q = 64, EMIT_G = 1024 / EMIT_Q;
__global__ __launch_bounds__(1024) void k_reach_emit(const uint16_t *__restrict__ u_hi,
                                                     const uint16_t *__restrict__ u_lo, int bp, int B,
                                                     const float *__restrict__ partial,
                                                     int n_parts, const int32_t *__restrict__ plan,
                                                     const int32_t *__restrict__ rows,
                                                     const int32_t *__restrict__ ext_of,
                                                     unsigned int *__restrict__ cnt,
                                                     unsigned long long *__restrict__ buf,
                                                     int64_t cap) {
    __shared__ float red[1024];
    griddep_wait();
    if (plan[0] == 0) return;
    const int nk = plan[1];
    const int qb_n = bp / EMIT_Q;
    const int i = blockIdx.x / qb_n;
    if (i >= nk) return;
    const int slot = plan[2 + i];
    const int b = (blockIdx.x % qb_n) * EMIT_Q + threadIdx.x % EMIT_Q;
    const int g = threadIdx.x / EMIT_Q;
    float acc = 0.f;
#pragma unroll 4
    for (int p = g; p < n_parts; p += EMIT_G) acc += partial[((int64_t)p * REACH_T + slot) * bp + b];
    red[threadIdx.x] = acc;
    __syncthreads();
    if (g == 0 && b < B) {
        float sum = red[threadIdx.x];
        for (int h = 1; h < EMIT_G; ++h) sum += red[h * EMIT_Q + threadIdx.x];
        const int64_t j = rows[slot];
        const float uj = __bfloat162float(__ushort_as_bfloat16(u_hi[j * bp + b])) +
                         __bfloat162float(__ushort_as_bfloat16(u_lo[j * bp + b]));
        const float s = uj + sum;
        buf[(int64_t)b * cap + i] = ((unsigned long long)__float_as_uint(s) << 32) |
                                    (unsigned long long)(~(uint32_t)ext_of[j]);
        if (i == 0) cnt[b] = (unsigned int)nk;
    }
}

int reach_parts() { return device_sm_count(); }

int64_t reach_pad_rows(int64_t n) { return (n + RM_BK - 1) / RM_BK * RM_BK; }


cudaError_t launch_reach_pack(const float *C, int64_t n, int H, float alpha, uint16_t *coef_hi,
                              uint16_t *coef_lo, cudaStream_t st) {
    const int64_t n_pad = reach_pad_rows(n);
    if (n_pad <= 0) return cudaSuccess;
    k_reach_pack<<<(unsigned)(n_pad / 64), 256, 0, st>>>(C, n, n_pad, H, alpha, coef_hi, coef_lo);
    return cudaGetLastError();
}

template <int BP>
static cudaError_t reach_mma_bp(const uint16_t *coef_hi, const uint16_t *coef_lo,
                                const uint16_t *u_hi, const uint16_t *u_lo, int64_t n,
                                const int32_t *plan, float *partial, int parts, int *status,
                                cudaStream_t st) {
    using C = RmCfg<BP>;
    static bool attr[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr[dev]) {
        cudaError_t e = cudaFuncSetAttribute(k_reach_mma<BP>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (e != cudaSuccess) return e;
        attr[dev] = true;
    }
    const int64_t n_pad = reach_pad_rows(n);
    CUtensorMap thi, tlo, thi64, tlo64;
    cudaError_t e = make_tmap_2d(&thi, coef_hi, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                                 (uint64_t)n_pad, RM_M, (uint64_t)n_pad * 2, RM_BK, RM_M);
    if (e == cudaSuccess)
        e = make_tmap_2d(&tlo, coef_lo, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (uint64_t)n_pad, RM_M,
                         (uint64_t)n_pad * 2, RM_BK, RM_M);
    if (e == cudaSuccess)
        e = make_tmap_2d(&thi64, coef_hi, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (uint64_t)n_pad,
                         RM_M, (uint64_t)n_pad * 2, RM_BK, RM_M / 2);
    if (e == cudaSuccess)
        e = make_tmap_2d(&tlo64, coef_lo, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (uint64_t)n_pad,
                         RM_M, (uint64_t)n_pad * 2, RM_BK, RM_M / 2);
    CUtensorMap tbh, tbl;
    if (e == cudaSuccess)
        e = make_tmap_2d(&tbh, u_hi, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, BP, (uint64_t)n,
                         (uint64_t)BP * 2, 64, RM_BK);
    if (e == cudaSuccess)
        e = make_tmap_2d(&tbl, u_lo, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, BP, (uint64_t)n,
                         (uint64_t)BP * 2, 64, RM_BK);
    if (e != cudaSuccess) return e;
    k_reach_mma<BP><<<parts, RM_THREADS, C::SMEM, st>>>(thi, tlo, thi64, tlo64, tbh, tbl, n, plan,
                                                         partial, status);
    return cudaGetLastError();
}

cudaError_t launch_reach_scores(const uint16_t *u_hi, const uint16_t *u_lo, int bp, int B,
                                int64_t n, const uint16_t *coef_hi,
                                const uint16_t *coef_lo, const int32_t *plan, const int32_t *rows,
                                const int32_t *ext_of, float *partial, unsigned int *cnt,
                                unsigned long long *buf, int64_t cap, int *status, cudaStream_t st,
                                int *launches) {
    if (n <= 0 || (bp != 128 && bp != 256)) return cudaErrorInvalidValue;
    const int parts = reach_parts();
    cudaError_t e = bp == 256 ? reach_mma_bp<256>(coef_hi, coef_lo, u_hi, u_lo, n, plan, partial,
                                                  parts, status, st)
                              : reach_mma_bp<128>(coef_hi, coef_lo, u_hi, u_lo, n, plan, partial,
                                                  parts, status, st);
    if (e != cudaSuccess) return e;
    e = launch_pdl(k_reach_emit, dim3(REACH_T * (bp / EMIT_Q)), dim3(1024), 0, st, u_hi, u_lo, bp, B,
                   (const float *)partial, parts, plan, rows, ext_of, cnt, buf, cap);
    if (launches) *launches += 2;
    return e == cudaSuccess ? cudaGetLastError() : e;
}

}  // namespace ak
