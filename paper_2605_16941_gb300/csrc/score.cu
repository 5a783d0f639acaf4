// score.cu -- fused LM-head GEMM + full-vocabulary softmax statistics (sm_103a).
//
// For every scored row h_n the method needs three numbers of the model's
// distribution p(. | Y~) = softmax_v(<h_n, w_v>) over the whole vocabulary
// (Eq. 2 and Eq. 3 of the WINO paper): argmax_v p, max_v p and p(target).
// The logits never leave the chip: each CTA pair computes 256 x bn logit
// tiles with 2-SM tensor-core MMAs (tcgen05.mma.cta_group::2, bf16 x bf16 ->
// fp32 in TMEM, M = 256 split 128/128 over the two SMs, N = bn <= 256), and four
// epilogue warps per CTA fold each tile straight out of TMEM into a running
// per-row state (max, sum of exp, argmax, target logit) that lives in
// registers across all of the pair's vocabulary tiles of that row block.  One
// partial record per (row, pair) goes to the workspace; finish.cu merges them.
//
// Kernel structure (persistent, clusters of 2 CTAs = one SM pair, 192 threads each):
//   warp 0  TMA producer (both CTAs): streams 64-wide K slices of its 128 rows
//           of H and of its bn/2 of the tile's bn W rows into a 6-stage ring;
//           both CTAs' copies complete on the LEADER's stage barrier;
//   warp 1  TMEM allocation (both CTAs, 512 columns = two 256-column fp32
//           accumulators) and, in the leader only, the MMA issuer:
//           4 x (M256 Nbn K16) per stage, committing stage release and
//           accumulator-ready to both CTAs (multicast);
//   warps 2-5 epilogue (both CTAs): one thread per row (TMEM lane); online
//           softmax over a tile's bn columns while the MMAs of the next tile
//           fill the other accumulator, then release the accumulator to the
//           leader's MMA warp (8 arrivals per tile).
// Work split: see ScoreArgs in internal.h.
//
// Every mbarrier wait is bounded (kWaitLimitNs): on expiry the CTA raises an
// abort flag and drains its in-flight copies and MMAs (again bounded); both
// CTAs then meet at the closing cluster barrier before TMEM is released, and
// the CTA records WINO_ERR_DEVICE_TIMEOUT in the call's status word.
//
// Optional timeline (ScoreArgs::timeline, diagnostics only): per CTA,
// globaltimer stamps [0] entry, [1] set-up done (barriers, TMEM), [2] first
// TMA issue, [3] griddepcontrol.wait returned in the epilogue, [4] last MMA
// completed (leader) or last tile read (peer), [5] all roles done, [6] exit;
// [7] = SM id << 32 | tiles of the pair.
#include <mutex>

#include "internal.h"
#include "ptx.cuh"
#include "wait.cuh"

namespace wino {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr uint16_t kBothCtas = 0x3;
constexpr int kPrefetchSlices = 16;  // K slices of the first tile prefetched into L2 before the grid wait

struct alignas(8) Barriers {
    uint64_t full[kStages];   // leader: both CTAs' copies of a stage landed
    uint64_t empty[kStages];  // both: the stage's MMAs are done (multicast commit)
    uint64_t tmem_full[2];    // both: accumulator i holds a finished tile (multicast commit)
    uint64_t tmem_empty[2];   // leader: all 8 epilogue warps of the pair have read accumulator i
    uint64_t mma_done;        // leader: every MMA issued has completed
    uint32_t tmem_base;
    int32_t abort;
};
static_assert(sizeof(Barriers) <= 256, "barrier block must fit its reserve");

template <bool kEntropy>
__global__ void __launch_bounds__(kScoreThreads, 1)
    score_kernel(const __grid_constant__ CUtensorMap tmH, const __grid_constant__ CUtensorMap tmW,
                 const ScoreArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_u32(smem_raw);
    const uint32_t ring = (raw + 1023u) & ~1023u;  // swizzle atoms need 1024-B alignment
    Barriers *bars = reinterpret_cast<Barriers *>(smem_raw + (ring - raw) + kRingBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = ptx::cluster_ctarank();  // 0: leader (issues the MMAs), 1: peer
    const bool leader = rank == 0;
    const int pair = blockIdx.x >> 1;
    uint64_t *const tl = a.timeline ? a.timeline + (size_t)blockIdx.x * kTimelineWords : nullptr;
    if (tl && threadIdx.x == 0)
        tl[0] = ptx::globaltimer_ns();

    auto sA = [&](int s) { return ring + (uint32_t)s * (kStageBytesA + kStageBytesB); };
    auto sB = [&](int s) { return sA(s) + kStageBytesA; };
    auto full = [&](int s) { return ptx::smem_u32(&bars->full[s]); };
    auto empty = [&](int s) { return ptx::smem_u32(&bars->empty[s]); };
    auto tfull = [&](int i) { return ptx::smem_u32(&bars->tmem_full[i]); };
    auto tempty = [&](int i) { return ptx::smem_u32(&bars->tmem_empty[i]); };
    const uint32_t mma_done = ptx::smem_u32(&bars->mma_done);

    // Set-up that touches no global memory overlaps the previous kernel (programmatic launch).
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(full(s), 1);
            ptx::mbar_init(empty(s), 1);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(tfull(i), 1);
            ptx::mbar_init(tempty(i), 8);  // 4 epilogue warps in each CTA of the pair
        }
        ptx::mbar_init(mma_done, 1);
        bars->abort = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        ptx::prefetch_tensormap(&tmH);
        ptx::prefetch_tensormap(&tmW);
    }
    if (warp == 1) {
        // Both CTAs of the pair take part in the pair allocation, which reserves the same columns in
        // both SMs; the address check below refuses to run if the two CTAs were given different ones.
        ptx::tmem_alloc_pair(ptx::smem_u32(&bars->tmem_base), kTmemCols);
        ptx::tmem_relinquish_pair();
    }
    ptx::tc_fence_before();
    ptx::cluster_sync();  // barriers and TMEM address of both CTAs are now visible to both
    ptx::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    const uint32_t peer_tmem = ptx::ld_shared_cluster_u32(ptx::mapa(ptx::smem_u32(&bars->tmem_base), rank ^ 1u));
    const bool tmem_ok = (peer_tmem == tmem);
    if (tl && threadIdx.x == 0)
        tl[1] = ptx::globaltimer_ns();

    // Programmatic launch: everything above overlapped the grid before us.  Whatever that grid is (the
    // previous WINO call's finish kernel, or a kernel of the caller's that wrote H), its writes are only
    // visible after griddepcontrol.wait, so every role waits before its first global access; the producer
    // first prefetches the start of its first tile into L2, which is safe before the wait (L2 is coherent).
    ptx::grid_dep_launch_dependents();

    const int grp = pair % a.n_groups;  // 256-row blocks grp, grp + n_groups, ...
    const int col = pair / a.n_groups;  // vocabulary tiles col, col + G, ...

    if (warp >= 2 || !tmem_ok) {
        ptx::grid_dep_wait();
        if (blockIdx.x == 0 && threadIdx.x == 64)
            a.status->finished = 0;  // the previous call's finish kernel has completed
        if (tl && threadIdx.x == 64)
            tl[3] = ptx::globaltimer_ns();
        for (int i = blockIdx.x * 128 + (int)threadIdx.x - 64; i < a.n_tickets; i += gridDim.x * 128)
            if (threadIdx.x >= 64)
                a.tickets[i] = 0;
    }
    if (!tmem_ok) {
        // nothing to do: the status word reports the failed allocation check
    } else if (warp == 0) {
        // ------------------------------------------------------------ TMA producer (both CTAs)
        const int half_bn = a.bn >> 1;  // W rows each CTA stages per tile
        if (lane == 0 && grp < a.n_mb && col < a.n_vt) {
            const int n_pre = min(a.n_kb, kPrefetchSlices);
            for (int kb = 0; kb < n_pre; ++kb) {
                ptx::tma_prefetch_2d(&tmW, kb * kBK, col * a.bn + (int)rank * half_bn);
                ptx::tma_prefetch_2d(&tmH, kb * kBK, grp * kPairM + (int)rank * kBM);
            }
        }
        ptx::grid_dep_wait();
        const uint64_t pol_h = ptx::policy_evict_last();    // H is re-read for every vocabulary tile
        const uint64_t pol_w = ptx::policy_evict_normal();  // W is shared by the row-block groups
        int stage = 0;
        uint32_t phase = 0;
        int32_t issued_parity[kStages];
        for (int s = 0; s < kStages; ++s)
            issued_parity[s] = -1;
        bool aborted = false;
        const uint32_t stage_tx = 2 * (kStageBytesA + (uint32_t)half_bn * (kBK * 2));  // both CTAs' copies
        bool first = true;
        for (int mb = grp; mb < a.n_mb && !aborted; mb += a.n_groups) {
            for (int vt = col; vt < a.n_vt && !aborted; vt += a.G) {
                for (int kb = 0; kb < a.n_kb; ++kb) {
                    int ok = 1;
                    if (lane == 0)
                        ok = wait_bounded(empty(stage), phase ^ 1u, &bars->abort);
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (!ok) {
                        aborted = true;
                        break;
                    }
                    if (lane == 0) {
                        const uint32_t bar = ptx::mapa(full(stage), 0);  // the leader's stage barrier
                        if (leader)
                            ptx::mbar_arrive_expect_tx(full(stage), stage_tx);
                        ptx::tma_load_2d_pair(sA(stage), &tmH, bar, kb * kBK, mb * kPairM + (int)rank * kBM, pol_h);
                        ptx::tma_load_2d_pair(sB(stage), &tmW, bar, kb * kBK, vt * a.bn + (int)rank * half_bn,
                                              pol_w);
                        if (tl && first)
                            tl[2] = ptx::globaltimer_ns();
                        first = false;
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
        if (aborted && leader && lane == 0) {
            // Let every copy already issued (by either CTA) land before the pair's shared memory goes away.
            for (int s = 0; s < kStages; ++s)
                if (issued_parity[s] >= 0)
                    wait_drain(full(s), (uint32_t)issued_parity[s]);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer (leader)
        if (leader) {
            const uint32_t idesc = ptx::idesc_bf16_f32(kPairM, (uint32_t)a.bn);
            int tiles = 0;
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool aborted = false;
            for (int mb = grp; mb < a.n_mb && !aborted; mb += a.n_groups) {
                for (int vt = col; vt < a.n_vt && !aborted; vt += a.G) {
                    int ok = 1;
                    if (lane == 0)
                        ok = wait_bounded<true>(tempty(acc), acc_phase ^ 1u, &bars->abort);
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
                            ok = wait_bounded(full(stage), phase, &bars->abort);
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
                                ptx::mma_bf16_pair(d_tmem, da + 2u * k, db + 2u * k, idesc, (kb | k) != 0);
                            ptx::mma_commit_pair_multicast(empty(stage), kBothCtas);
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
                        ptx::mma_commit_pair_multicast(tfull(acc), kBothCtas);
                    __syncwarp();
                    ++tiles;
                    if (++acc == 2) {
                        acc = 0;
                        acc_phase ^= 1u;
                    }
                }
            }
            // No MMA may still be writing either CTA's TMEM when it is released.
            if (lane == 0) {
                ptx::mma_commit_pair(mma_done);
                wait_drain(mma_done, 0);
                if (tl) {
                    tl[4] = ptx::globaltimer_ns();
                    tl[7] = (uint64_t)ptx::smid() << 32 | (uint32_t)tiles;
                }
            }
            __syncwarp();
        }
    } else {
        // ------------------------------------------------------------ epilogue (warps 2..5, both CTAs)
        const int q = warp & 3;  // this warp may only read TMEM lanes [32q, 32q + 32)
        int acc = 0;
        uint32_t acc_phase = 0;
        bool aborted = false;
        for (int mb = grp; mb < a.n_mb && !aborted; mb += a.n_groups) {
            const int64_t row = (int64_t)mb * kPairM + (int)rank * kBM + q * 32 + lane;
            const int32_t tgt = (row < a.N) ? row_target(a.ts, row, a.V) : -1;
            float m = -INFINITY, s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f, tlog = -INFINITY;
            float u0 = 0.f, u1 = 0.f, u2 = 0.f, u3 = 0.f;  // entropy variant
            int32_t am = 0;
            for (int vt = col; vt < a.n_vt; vt += a.G) {
                const int32_t v0 = vt * a.bn;
                const int nvalid = min(a.bn, a.V - v0);
                int ok = 1;
                if (lane == 0)
                    ok = wait_bounded(tfull(acc), acc_phase, &bars->abort);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) {
                    aborted = true;
                    break;
                }
                ptx::tc_fence_after();
                const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kBN);
#pragma unroll 1
                for (int c = 0; c < kBN / 32; ++c) {
                    const int cvalid = nvalid - c * 32;  // warp-uniform; columns past the tile are masked
                    if (cvalid <= 0)
                        break;
                    float x[32];
                    ptx::tmem_ld_32x32b_x32(tbase + (uint32_t)(c * 32), x);
                    ptx::tmem_ld_wait();
                    if (cvalid < 32) {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (j >= cvalid)
                                x[j] = -INFINITY;  // past V (TMA zero fill) or past the tile (another tile's columns)
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
                        if (kEntropy && m != -INFINITY) {  // u' = scale * (u + (m - cm) log2(e) * s)
                            const float dl = (m - cm) * kLog2e;
                            u0 = scale * fmaf(dl, s0, u0);
                            u1 = scale * fmaf(dl, s1, u1);
                            u2 = scale * fmaf(dl, s2, u2);
                            u3 = scale * fmaf(dl, s3, u3);
                        }
                        s0 *= scale;
                        s1 *= scale;
                        s2 *= scale;
                        s3 *= scale;
                        m = cm;
                    }
                    const float mb2 = m * kLog2e;
                    if (!kEntropy) {
#pragma unroll
                        for (int j = 0; j < 32; j += 4) {
                            s0 += ptx::ex2(fmaf(x[j + 0], kLog2e, -mb2));
                            s1 += ptx::ex2(fmaf(x[j + 1], kLog2e, -mb2));
                            s2 += ptx::ex2(fmaf(x[j + 2], kLog2e, -mb2));
                            s3 += ptx::ex2(fmaf(x[j + 3], kLog2e, -mb2));
                        }
                    } else {
                        // t = (l - m) log2(e), kept finite (masked columns are -inf; 2^-200 is 0 in fp32 anyway)
#pragma unroll
                        for (int j = 0; j < 32; j += 4) {
                            const float t0 = fmaxf(fmaf(x[j + 0], kLog2e, -mb2), -200.f);
                            const float t1 = fmaxf(fmaf(x[j + 1], kLog2e, -mb2), -200.f);
                            const float t2 = fmaxf(fmaf(x[j + 2], kLog2e, -mb2), -200.f);
                            const float t3 = fmaxf(fmaf(x[j + 3], kLog2e, -mb2), -200.f);
                            const float e0 = ptx::ex2(t0), e1 = ptx::ex2(t1), e2 = ptx::ex2(t2), e3 = ptx::ex2(t3);
                            s0 += e0;
                            s1 += e1;
                            s2 += e2;
                            s3 += e3;
                            u0 = fmaf(e0, t0, u0);
                            u1 = fmaf(e1, t1, u1);
                            u2 = fmaf(e2, t2, u2);
                            u3 = fmaf(e3, t3, u3);
                        }
                    }
                    const int tj = tgt - (v0 + c * 32);
                    if ((unsigned)tj < 32u) {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            tlog = (j == tj) ? x[j] : tlog;
                    }
                }
                // Accumulator fully read by this warp: tell the leader's MMA warp.
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    ptx::mbar_arrive_cluster(ptx::mapa(tempty(acc), 0));
                if (++acc == 2) {
                    acc = 0;
                    acc_phase ^= 1u;
                }
            }
            if (!aborted && row < a.N) {
                a.part[row * a.G + col] = make_float4(m, (s0 + s1) + (s2 + s3), __int_as_float(am), tlog);
                if (kEntropy)
                    a.part_u[row * a.G + col] = (u0 + u1) + (u2 + u3);
            }
        }
        if (tl && !leader && warp == 2 && lane == 0)
            tl[4] = ptx::globaltimer_ns();
    }

    // Neither CTA releases TMEM, or exits, while its peer may still use the pair's TMEM or barriers.
    ptx::tc_fence_before();
    __syncthreads();
    if (tl && threadIdx.x == 0)
        tl[5] = ptx::globaltimer_ns();
    if (threadIdx.x == 64) {
        // Warp 2 has passed griddepcontrol.wait, so the previous call's finish kernel, which clears the
        // status word, has completed: a failure recorded now belongs to this call.
        if (!tmem_ok)
            atomicExch(&a.status->current, (int32_t)WINO_ERR_UNSUPPORTED);
        else if (*reinterpret_cast<volatile int32_t *>(&bars->abort))
            atomicExch(&a.status->current, (int32_t)WINO_ERR_DEVICE_TIMEOUT);
    }
    ptx::cluster_sync();
    ptx::tc_fence_after();
    if (warp == 1)
        ptx::tmem_dealloc_pair(tmem, kTmemCols);
    if (tl && threadIdx.x == 0)
        tl[6] = ptx::globaltimer_ns();
}

}  // namespace

// Choose the tile width bn and the number of row-block groups: fewest vocabulary columns on the busiest
// pair (tiles x (bn + a per-tile overhead)), then the widest tile, then fewest passes over W (more groups).
// A width below kBN pays when the vocabulary then splits evenly over the pairs: V = 126464 on 76 pairs is
// 494 tiles of 256 (7 on the busiest pair, 6.5 on average) but 527 tiles of 240 (7 on the busiest pair).
ScoreSchedule score_schedule(int32_t n_mb, int64_t V, int max_units, int32_t records_cap)
{
    constexpr int64_t kTileOverheadCols = 16;  // H re-read and accumulator hand-over per tile, in columns
    ScoreSchedule best{kBN, (int32_t)((V + kBN - 1) / kBN), 1, 1};
    int64_t best_cost = -1;
    const int32_t top = n_mb < max_units ? n_mb : max_units;
    for (int32_t bn = kBN; bn >= kMinBN; bn -= 16) {
        const int64_t n_vt = (V + bn - 1) / bn;
        for (int32_t groups = top; groups >= 1; --groups) {
            int64_t g = max_units / groups;
            g = g < n_vt ? g : n_vt;
            g = g < records_cap ? g : records_cap;
            g = g < kMaxRecordsPerRow ? g : kMaxRecordsPerRow;
            g = g < 1 ? 1 : g;
            const int64_t rounds = (int64_t)((n_mb + groups - 1) / groups) * ((n_vt + g - 1) / g);
            const int64_t cost = rounds * (bn + kTileOverheadCols);
            if (best_cost < 0 || cost < best_cost) {
                best_cost = cost;
                best = ScoreSchedule{bn, (int32_t)n_vt, groups, (int32_t)g};
            }
        }
    }
    return best;
}

namespace {

cudaLaunchConfig_t score_config(unsigned grid, cudaStream_t stream, cudaLaunchAttribute (&attr)[2])
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kScoreThreads);
    cfg.dynamicSmemBytes = kScoreSmemBytes;
    cfg.stream = stream;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cfg;
}

// Per-device one-time set-up: shared-memory opt-in and the number of co-resident pairs.
int configure_device()
{
    static std::mutex mu;
    static int pairs[64];
    static bool done[64];
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64)
        return -1;
    std::lock_guard<std::mutex> g(mu);
    if (!done[dev]) {
        if (cudaFuncSetAttribute(score_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kScoreSmemBytes) != cudaSuccess ||
            cudaFuncSetAttribute(score_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kScoreSmemBytes) != cudaSuccess)
            return -1;
        cudaLaunchAttribute attr[2];
        cudaLaunchConfig_t cfg = score_config(2, nullptr, attr);
        cfg.numAttrs = 1;  // the cluster shape is what matters for the occupancy query
        int clusters = 0;
        if (cudaOccupancyMaxActiveClusters(&clusters, score_kernel<false>, &cfg) != cudaSuccess || clusters < 1)
            return -1;
        pairs[dev] = clusters;
        done[dev] = true;
    }
    return pairs[dev];
}

}  // namespace

int score_max_pairs() { return configure_device(); }

cudaError_t launch_score(const CUtensorMap &tmH, const CUtensorMap &tmW, const ScoreArgs &a, bool entropy,
                         cudaStream_t stream)
{
    if (configure_device() < 1)
        return cudaErrorUnknown;
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = score_config((unsigned)(2 * a.n_groups * a.G), stream, attr);
    return entropy ? cudaLaunchKernelEx(&cfg, score_kernel<true>, tmH, tmW, a)
                   : cudaLaunchKernelEx(&cfg, score_kernel<false>, tmH, tmW, a);
}

}  // namespace wino
