// score.cu -- fused LM-head GEMM + full-vocabulary softmax statistics (sm_103a).
//
// For every scored row h_n the method needs three numbers of the model's
// distribution p(. | Y~) = softmax_v(<h_n, w_v>) over the whole vocabulary
// (Eq. 2 and Eq. 3 of the WINO paper): argmax_v p, max_v p and p(target).
// The logits never leave the chip: each CTA computes 128 x 256 logit tiles
// on the tensor cores (tcgen05.mma, bf16 x bf16 -> fp32 in TMEM), and four
// epilogue warps fold each tile straight out of TMEM into a running
// per-row state (max, sum of exp, argmax, target logit) that lives in
// registers across all of the CTA's vocabulary tiles of that row block.  One
// partial record per (row, CTA) goes to the workspace; finish.cu merges them.
//
// Kernel structure (persistent, one CTA per SM, 192 threads):
//   warp 0  TMA producer: streams 64-wide K slices of H (128 rows) and W
//           (256 vocabulary rows) into a 4-stage shared-memory ring;
//   warp 1  MMA issuer: allocates 512 TMEM columns (two 256-column fp32
//           accumulators), issues 4 x (M128 N256 K16) MMAs per stage and
//           commits stage-release / accumulator-ready barriers;
//   warps 2-5 epilogue: one thread per row (TMEM lane), online softmax over
//           each tile's 256 columns while the MMA warp fills the other
//           accumulator.
// Work split: see ScoreArgs in internal.h (row-block groups walking the
// vocabulary side by side).
//
// Every mbarrier wait is bounded (kWaitLimitNs): on expiry the CTA raises an
// abort flag, records WINO_ERR_DEVICE_TIMEOUT in the status word, drains its
// in-flight copies and MMAs (again bounded) and frees its TMEM.
#include "internal.h"
#include "ptx.cuh"

namespace wino {
namespace {

constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s per wait
constexpr uint64_t kDrainLimitNs = 200000000ull;   // 0.2 s for draining after an abort
constexpr float kLog2e = 1.4426950408889634f;

struct alignas(8) Barriers {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t tmem_full[2];
    uint64_t tmem_empty[2];
    uint64_t mma_done;
    uint32_t tmem_base;
    int32_t abort;
};
static_assert(sizeof(Barriers) <= 256, "barrier block must fit its reserve");

// Wait for phase `parity` of `bar`; false once the wait limit passed or another
// role of this CTA aborted.
__device__ bool wait_bounded(uint32_t bar, uint32_t parity, int32_t *abort_flag, int32_t *status)
{
    if (ptx::mbar_try_wait(bar, parity))
        return true;
    const uint64_t t0 = ptx::globaltimer_ns();
    for (uint32_t it = 1;; ++it) {
        if (ptx::mbar_try_wait(bar, parity))
            return true;
        if ((it & 15u) == 0) {
            if (*reinterpret_cast<volatile int32_t *>(abort_flag))
                return false;
            if (ptx::globaltimer_ns() - t0 > kWaitLimitNs) {
                atomicExch(abort_flag, 1);
                atomicExch(status, (int32_t)WINO_ERR_DEVICE_TIMEOUT);
                return false;
            }
        }
    }
}

// Bounded wait that ignores the abort flag (used only to drain after an abort).
__device__ bool wait_drain(uint32_t bar, uint32_t parity)
{
    const uint64_t t0 = ptx::globaltimer_ns();
    while (!ptx::mbar_try_wait(bar, parity))
        if (ptx::globaltimer_ns() - t0 > kDrainLimitNs)
            return false;
    return true;
}

__global__ void __launch_bounds__(kScoreThreads, 1)
    score_kernel(const __grid_constant__ CUtensorMap tmH, const __grid_constant__ CUtensorMap tmW,
                 const ScoreArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_u32(smem_raw);
    const uint32_t ring = (raw + 1023u) & ~1023u;  // swizzle atoms need 1024-B alignment
    Barriers *bars = reinterpret_cast<Barriers *>(smem_raw + (ring - raw) + kRingBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    auto sA = [&](int s) { return ring + (uint32_t)s * (kStageBytesA + kStageBytesB); };
    auto sB = [&](int s) { return sA(s) + kStageBytesA; };
    auto full = [&](int s) { return ptx::smem_u32(&bars->full[s]); };
    auto empty = [&](int s) { return ptx::smem_u32(&bars->empty[s]); };
    auto tfull = [&](int s) { return ptx::smem_u32(&bars->tmem_full[s]); };
    auto tempty = [&](int s) { return ptx::smem_u32(&bars->tmem_empty[s]); };

    // Set-up that touches no global memory overlaps the previous kernel (programmatic launch).
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(full(s), 1);
            ptx::mbar_init(empty(s), 1);
        }
        for (int s = 0; s < 2; ++s) {
            ptx::mbar_init(tfull(s), 1);
            ptx::mbar_init(tempty(s), 4);  // one arrival per epilogue warp
        }
        ptx::mbar_init(ptx::smem_u32(&bars->mma_done), 1);
        bars->abort = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        ptx::prefetch_tensormap(&tmH);
        ptx::prefetch_tensormap(&tmW);
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_u32(&bars->tmem_base), kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;

    // From here on global memory is read and written: wait for the grid before us.
    ptx::grid_dep_wait();
    ptx::grid_dep_launch_dependents();
    if (blockIdx.x == 0 && threadIdx.x == 0)
        *a.status = WINO_OK;  // a timeout, if any, is raised no earlier than kWaitLimitNs later
    for (int i = blockIdx.x * kScoreThreads + threadIdx.x; i < a.n_tickets; i += gridDim.x * kScoreThreads)
        a.tickets[i] = 0;

    const int grp = blockIdx.x % a.n_groups;  // row blocks grp, grp + n_groups, ...
    const int col = blockIdx.x / a.n_groups;  // vocabulary tiles col, col + G, ...

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        const uint64_t pol_h = ptx::policy_evict_last();    // H is re-read for every vocabulary tile
        const uint64_t pol_w = ptx::policy_evict_normal();  // W is shared by the row-block groups
        int stage = 0;
        uint32_t phase = 0;
        int32_t issued_parity[kStages];
        for (int s = 0; s < kStages; ++s)
            issued_parity[s] = -1;
        bool aborted = false;
        for (int mb = grp; mb < a.n_mb && !aborted; mb += a.n_groups) {
            for (int vt = col; vt < a.n_vt && !aborted; vt += a.G) {
                for (int kb = 0; kb < a.n_kb; ++kb) {
                    int ok = 1;
                    if (lane == 0)
                        ok = wait_bounded(empty(stage), phase ^ 1u, &bars->abort, a.status);
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (!ok) {
                        aborted = true;
                        break;
                    }
                    if (lane == 0) {
                        ptx::mbar_arrive_expect_tx(full(stage), kStageBytesA + kStageBytesB);
                        ptx::tma_load_2d(sA(stage), &tmH, full(stage), kb * kBK, mb * kBM, pol_h);
                        ptx::tma_load_2d(sB(stage), &tmW, full(stage), kb * kBK, vt * kBN, pol_w);
                    }
                    __syncwarp();
                    issued_parity[stage] = (int32_t)phase;
                    if (++stage == kStages) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
        }
        if (aborted && lane == 0) {
            // Let every copy already issued land before the CTA (and its shared memory) goes away.
            for (int s = 0; s < kStages; ++s)
                if (issued_parity[s] >= 0)
                    wait_drain(full(s), (uint32_t)issued_parity[s]);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        constexpr uint32_t idesc = ptx::idesc_bf16_f32(kBM, kBN);
        int stage = 0;
        uint32_t phase = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        bool aborted = false;
        for (int mb = grp; mb < a.n_mb && !aborted; mb += a.n_groups) {
            for (int vt = col; vt < a.n_vt && !aborted; vt += a.G) {
                int ok = 1;
                if (lane == 0)
                    ok = wait_bounded(tempty(acc), acc_phase ^ 1u, &bars->abort, a.status);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) {
                    aborted = true;
                    break;
                }
                ptx::tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(acc * kBN);
                for (int kb = 0; kb < a.n_kb; ++kb) {
                    ok = 1;
                    if (lane == 0)
                        ok = wait_bounded(full(stage), phase, &bars->abort, a.status);
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (!ok) {
                        aborted = true;
                        break;
                    }
                    ptx::tc_fence_after();
                    if (lane == 0) {
                        const uint64_t da = ptx::sdesc_kmajor_sw128(sA(stage));
                        const uint64_t db = ptx::sdesc_kmajor_sw128(sB(stage));
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k)  // +32 B along K per MMA = +2 in the encoded address
                            ptx::mma_bf16(d_tmem, da + 2u * k, db + 2u * k, idesc, (kb | k) != 0);
                        ptx::mma_commit(empty(stage));
                    }
                    __syncwarp();
                    if (++stage == kStages) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (aborted)
                    break;
                if (lane == 0)
                    ptx::mma_commit(tfull(acc));
                __syncwarp();
                if (++acc == 2) {
                    acc = 0;
                    acc_phase ^= 1u;
                }
            }
        }
        // No MMA may still be writing TMEM when it is released.
        if (lane == 0) {
            ptx::mma_commit(ptx::smem_u32(&bars->mma_done));
            wait_drain(ptx::smem_u32(&bars->mma_done), 0);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue (warps 2..5)
        const int q = warp & 3;  // this warp may only read TMEM lanes [32q, 32q + 32)
        int acc = 0;
        uint32_t acc_phase = 0;
        bool aborted = false;
        for (int mb = grp; mb < a.n_mb && !aborted; mb += a.n_groups) {
            const int64_t row = (int64_t)mb * kBM + q * 32 + lane;
            const int32_t tgt = (row < a.N) ? row_target(a.ts, row, a.V) : -1;
            float m = -INFINITY, s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f, tl = 0.f;
            int32_t am = 0;
            for (int vt = col; vt < a.n_vt; vt += a.G) {
                const int32_t v0 = vt * kBN;
                const int nvalid = min(kBN, a.V - v0);
                int ok = 1;
                if (lane == 0)
                    ok = wait_bounded(tfull(acc), acc_phase, &bars->abort, a.status);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) {
                    aborted = true;
                    break;
                }
                ptx::tc_fence_after();
                const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kBN);
#pragma unroll 1
                for (int c = 0; c < kBN / 32; ++c) {
                    const int cvalid = nvalid - c * 32;  // warp-uniform
                    if (cvalid <= 0)
                        break;
                    float x[32];
                    ptx::tmem_ld_32x32b_x32(tbase + (uint32_t)(c * 32), x);
                    ptx::tmem_ld_wait();
                    if (cvalid < 32) {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (j >= cvalid)
                                x[j] = -INFINITY;  // columns past V are TMA zero fill, not logits
                    }
                    float cm = x[0];
#pragma unroll
                    for (int j = 1; j < 32; ++j)
                        cm = fmaxf(cm, x[j]);
                    if (cm > m) {  // strict: an earlier column keeps the argmax on ties
                        int j0 = 31;
#pragma unroll
                        for (int j = 31; j >= 0; --j)
                            if (x[j] == cm)
                                j0 = j;
                        am = v0 + c * 32 + j0;
                        const float scale = ptx::ex2((m - cm) * kLog2e);
                        s0 *= scale;
                        s1 *= scale;
                        s2 *= scale;
                        s3 *= scale;
                        m = cm;
                    }
                    const float mb2 = m * kLog2e;
#pragma unroll
                    for (int j = 0; j < 32; j += 4) {
                        s0 += ptx::ex2(fmaf(x[j + 0], kLog2e, -mb2));
                        s1 += ptx::ex2(fmaf(x[j + 1], kLog2e, -mb2));
                        s2 += ptx::ex2(fmaf(x[j + 2], kLog2e, -mb2));
                        s3 += ptx::ex2(fmaf(x[j + 3], kLog2e, -mb2));
                    }
                    const int tj = tgt - (v0 + c * 32);
                    if ((unsigned)tj < 32u) {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            tl = (j == tj) ? x[j] : tl;
                    }
                }
                // Accumulator fully read: hand it back to the MMA warp.
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    ptx::mbar_arrive(tempty(acc));
                if (++acc == 2) {
                    acc = 0;
                    acc_phase ^= 1u;
                }
            }
            if (!aborted && row < a.N)
                a.part[row * a.G + col] = make_float4(m, (s0 + s1) + (s2 + s3), __int_as_float(am), tl);
        }
        ptx::tc_fence_before();
    }

    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

// Choose the number of row-block groups: fewest tiles on the busiest CTA,
// then fewest passes over W (more groups = fewer passes).
void score_schedule(int32_t n_mb, int32_t n_vt, int max_ctas, int32_t *n_groups, int32_t *G)
{
    int64_t best_rounds = -1;
    int32_t best_groups = 1, best_g = 1;
    const int32_t top = n_mb < max_ctas ? n_mb : max_ctas;
    for (int32_t groups = top; groups >= 1; --groups) {
        int32_t g = max_ctas / groups;
        g = g < n_vt ? g : n_vt;
        g = g < kMaxRecordsPerRow ? g : kMaxRecordsPerRow;
        g = g < 1 ? 1 : g;
        const int64_t rounds = (int64_t)((n_mb + groups - 1) / groups) * ((n_vt + g - 1) / g);
        if (best_rounds < 0 || rounds < best_rounds) {
            best_rounds = rounds;
            best_groups = groups;
            best_g = g;
        }
    }
    *n_groups = best_groups;
    *G = best_g;
}

cudaError_t launch_score(const CUtensorMap &tmH, const CUtensorMap &tmW, const ScoreArgs &a, cudaStream_t stream)
{
    static thread_local int configured_device = -1;
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    if (configured_device != dev) {
        e = cudaFuncSetAttribute(score_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kScoreSmemBytes);
        if (e != cudaSuccess)
            return e;
        configured_device = dev;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(a.n_groups * a.G));
    cfg.blockDim = dim3(kScoreThreads);
    cfg.dynamicSmemBytes = kScoreSmemBytes;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, score_kernel, tmH, tmW, a);
}

}  // namespace wino
