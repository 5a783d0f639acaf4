// score.cu -- fused LM-head GEMM + full-vocabulary softmax statistics (sm_103a).
//
// For every scored row h_n the method needs three numbers of the model's
// distribution p(. | Y~) = softmax_v(<h_n, w_v>) over the whole vocabulary
// (Eq. 2 and Eq. 3 of the WINO paper): argmax_v p, max_v p and p(target).
// The logits never leave the chip: each CTA pair computes logit tiles of 256
// rows x bn vocabulary columns with 2-SM tensor-core MMAs
// (tcgen05.mma.cta_group::2, bf16 x bf16 -> fp32 in TMEM, M = 256 split
// 128/128 over the two SMs, N = bn <= 256), and four epilogue warps per CTA
// fold each tile straight out of TMEM into a running per-row state (max, sum
// of exp, argmax, target logit) that lives in registers across all of the
// pair's vocabulary tiles of that row block.  One partial record per
// (row, pair) goes to the workspace; finish.cu merges them.
//
// Two modes (ScoreArgs::two, chosen per launch by score_schedule):
//   single tiles, for shapes bound by the W stream from HBM (one 256-row
//     block): the two accumulators alternate between consecutive tiles, so
//     the epilogue of one tile overlaps the MMAs of the next, and the ring has
//     up to 7 stages, the most W bytes in flight per SM;
//   passes, for tensor-bound shapes: a stage holds three 16 KB slots and
//     feeds both accumulators, a quarter fewer bytes delivered per SM and MMA
//     than single tiles.  A group of pairs that owns two or more row blocks
//     takes them two at a time (row-pair sweeps): the two blocks' H slices
//     and one tile's W slice, so every W slice staged serves both blocks and
//     the group streams W from HBM once per two blocks.  A block left without
//     a partner is swept alone (tile-pair sweeps): its H slice and the slices
//     of two tiles.  The accumulators then fill TMEM, so a pass's MMAs into
//     the first accumulator start as soon as the epilogue has read it, and
//     its MMAs into the second accumulator for the first ring stages are
//     deferred until the epilogue has read that one too (the stages are
//     released after those).
//
// Kernel structure (persistent, clusters of 2 CTAs = one SM pair, 192 threads each):
//   warp 0  TMA producer (both CTAs): per K slice, its 128 rows of H (of one
//           or two row blocks) and its bn/2 of the (one or two) tiles' W rows
//           into the ring; both CTAs' copies complete on the LEADER's stage
//           barrier;
//   warp 1  TMEM allocation (both CTAs, all 512 columns) and, in the leader
//           only, the MMA issuer: 4 x (M256 Nbn K16) per stage and tile,
//           committing stage release and accumulator-ready to both CTAs
//           (multicast);
//   warps 2-5 epilogue (both CTAs): one thread per row (TMEM lane); online
//           softmax over a tile's columns, then release of the accumulator to
//           the leader's MMA warp (8 arrivals per accumulator use).
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
constexpr int kPrefetchSlices = 4;   // K slices of the first W tile prefetched into L2 before the grid wait
constexpr int kTmemLoadsPerWait = 1;  // 32-column TMEM loads in flight per tcgen05.wait::ld in the epilogue (2 measured slower)

struct alignas(8) Barriers {
    uint64_t full[kMaxStages];   // leader: both CTAs' copies of a stage landed
    uint64_t empty[kMaxStages];  // both: the stage's MMAs are done (multicast commit)
    uint64_t tmem_full[2];       // both: accumulator i holds a finished tile (multicast commit)
    uint64_t tmem_empty[2];      // leader: all 8 epilogue warps of the pair have read accumulator i
    uint64_t mma_done;           // leader: every MMA issued has completed
    uint32_t tmem_base;
    int32_t abort;
};
static_assert(sizeof(Barriers) <= 256, "barrier block must fit its reserve");

// Running softmax state of one row (one thread), across all of a pair's tiles of that row.
struct RowState {
    float m, s0, s1, s2, s3, tlog;
    float u0, u1, u2, u3;  // entropy variant: sum of exp(l - m) (l - m) log2(e)
    int32_t am;
};

// Fold 32 consecutive logits x (columns v .. v + 31; those at or past cvalid are not logits) into the row
// state: online max with rescaling, four partial sums of 2^((l - m) log2 e), argmax (an earlier column
// keeps it on ties), and the target's logit when it lies among them.
template <bool kEntropy>
__device__ __forceinline__ void fold32(RowState &r, float (&x)[32], int v, int cvalid, int tgt)
{
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
    if (cm > r.m) {  // strict: an earlier column keeps the argmax on ties
        int j0 = 31;
#pragma unroll
        for (int j = 31; j >= 0; --j)
            if (x[j] == cm)
                j0 = j;
        r.am = v + j0;
        const float scale = ptx::ex2((r.m - cm) * kLog2e);
        if (kEntropy && r.m != -INFINITY) {  // u' = scale * (u + (m - cm) log2(e) * s)
            const float dl = (r.m - cm) * kLog2e;
            r.u0 = scale * fmaf(dl, r.s0, r.u0);
            r.u1 = scale * fmaf(dl, r.s1, r.u1);
            r.u2 = scale * fmaf(dl, r.s2, r.u2);
            r.u3 = scale * fmaf(dl, r.s3, r.u3);
        }
        r.s0 *= scale;
        r.s1 *= scale;
        r.s2 *= scale;
        r.s3 *= scale;
        r.m = cm;
    }
    const float mb2 = r.m * kLog2e;
    if (!kEntropy) {
#pragma unroll
        for (int j = 0; j < 32; j += 4) {
            r.s0 += ptx::ex2(fmaf(x[j + 0], kLog2e, -mb2));
            r.s1 += ptx::ex2(fmaf(x[j + 1], kLog2e, -mb2));
            r.s2 += ptx::ex2(fmaf(x[j + 2], kLog2e, -mb2));
            r.s3 += ptx::ex2(fmaf(x[j + 3], kLog2e, -mb2));
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
            r.s0 += e0;
            r.s1 += e1;
            r.s2 += e2;
            r.s3 += e3;
            r.u0 = fmaf(e0, t0, r.u0);
            r.u1 = fmaf(e1, t1, r.u1);
            r.u2 = fmaf(e2, t2, r.u2);
            r.u3 = fmaf(e3, t3, r.u3);
        }
    }
    const int tj = tgt - v;
    if ((unsigned)tj < 32u) {
#pragma unroll
        for (int j = 0; j < 32; ++j)
            r.tlog = (j == tj) ? x[j] : r.tlog;
    }
}

// Fold the nvalid first columns of one accumulator (this warp's 32 TMEM lanes from tbase), vocabulary
// ids v0 ..; kTmemLoadsPerWait 32-column loads in flight per wait.
template <bool kEntropy>
__device__ __forceinline__ void fold_tile(RowState &r, uint32_t tbase, int v0, int nvalid, int tgt)
{
#pragma unroll 1
    for (int c = 0; c * 32 < nvalid; c += kTmemLoadsPerWait) {
        float x[kTmemLoadsPerWait][32];
#pragma unroll
        for (int i = 0; i < kTmemLoadsPerWait; ++i)
            if (i == 0 || (c + i) * 32 < nvalid)  // warp-uniform
                ptx::tmem_ld_32x32b_x32(tbase + (uint32_t)((c + i) * 32), x[i]);
        ptx::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < kTmemLoadsPerWait; ++i)
            if (i == 0 || (c + i) * 32 < nvalid)
                fold32<kEntropy>(r, x[i], v0 + (c + i) * 32, nvalid - (c + i) * 32, tgt);
    }
}

// kTwo: passes (ScoreArgs::two == 1: row-pair and tile-pair sweeps), else single tiles.
template <bool kEntropy, bool kTwo>
__global__ void __launch_bounds__(kScoreThreads, 1)
    score_kernel(const __grid_constant__ CUtensorMap tmH, const __grid_constant__ CUtensorMap tmW,
                 const ScoreArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_u32(smem_raw);
    const uint32_t ring = (raw + 1023u) & ~1023u;  // swizzle atoms need 1024-B alignment
    Barriers *bars = reinterpret_cast<Barriers *>(smem_raw + (ring - raw) + (uint32_t)a.stages * a.stage_bytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = ptx::cluster_ctarank();  // 0: leader (issues the MMAs), 1: peer
    const bool leader = rank == 0;
    const int pair = blockIdx.x >> 1;
    uint64_t *const tl = a.timeline ? a.timeline + (size_t)blockIdx.x * kTimelineWords : nullptr;
    // The records of an epilogue thread's last sweep (one row, or two in a row-pair sweep) are stored after
    // this CTA's arrival on the closing cluster barrier, so that the barrier's release does not wait for them.
    float4 pend[2] = {make_float4(0.f, 0.f, 0.f, 0.f), make_float4(0.f, 0.f, 0.f, 0.f)};
    float pend_u[2] = {0.f, 0.f};
    int64_t pend_idx[2] = {-1, -1};
    if (tl && threadIdx.x == 0)
        tl[0] = ptx::globaltimer_ns();

    const int S = a.stages;
    const uint32_t wb = stage_bytes_w(a.bn);
    auto sA = [&](int s) { return ring + (uint32_t)s * a.stage_bytes; };
    auto sB = [&](int s, int t) { return sA(s) + kStageBytesA + (uint32_t)t * wb; };
    auto full = [&](int s) { return ptx::smem_u32(&bars->full[s]); };
    auto empty = [&](int s) { return ptx::smem_u32(&bars->empty[s]); };
    auto tfull = [&](int i) { return ptx::smem_u32(&bars->tmem_full[i]); };
    auto tempty = [&](int i) { return ptx::smem_u32(&bars->tmem_empty[i]); };
    const uint32_t mma_done = ptx::smem_u32(&bars->mma_done);

    // Set-up that touches no global memory overlaps the previous kernel (programmatic launch).
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
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
    // first prefetches the start of its first W tile into L2, which is safe before the wait (L2 is coherent).
    ptx::grid_dep_launch_dependents();

    const int grp = pair % a.n_groups;  // 256-row blocks grp, grp + n_groups, ...
    const int col = pair / a.n_groups;  // vocabulary tiles col, col + G, ...
    // Sweeps over the pair's vocabulary tiles.  Single tiles: one sweep per row block, one tile per item.
    // Passes: row blocks mb and mb + n_groups together (row-pair sweep: item = one tile of both blocks, so
    // each W slice staged serves both and the group reads W once per two blocks), or a block left without
    // a partner alone (tile-pair sweep: item = tiles vt and vt + G of that block).
    const int mb_step = kTwo ? 2 * a.n_groups : a.n_groups;
    const int vstep = kTwo ? 2 * a.G : a.G;  // tiles per item of a single-tile or tile-pair sweep

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
        // W map coordinates of (K slice kb, vocabulary row v): (64 kb, v) in row-major W, (0, kb V + v) in the
        // panel copy
        auto w_x = [&](int kb) { return a.w_panels ? 0 : kb * kBK; };
        auto w_y = [&](int kb, int v) { return a.w_panels ? kb * a.V + v : v; };
        if (lane == 0 && grp < a.n_mb)
            for (int kb = 0; kb < min(a.n_kb, kPrefetchSlices); ++kb)
                ptx::tma_prefetch_2d(&tmW, w_x(kb), w_y(kb, col * a.bn + (int)rank * half_bn));
        ptx::grid_dep_wait();
        const uint64_t pol_h = ptx::policy_evict_last();    // H is re-read for every item
        const uint64_t pol_w = ptx::policy_evict_normal();  // W is shared by the row-block groups
        int stage = 0;
        uint32_t phase = 0;
        int32_t issued_parity[kMaxStages];
        for (int s = 0; s < kMaxStages; ++s)
            issued_parity[s] = -1;
        bool aborted = false;
        bool first = true;
        for (int mb = grp; mb < a.n_mb && !aborted; mb += mb_step) {
            const int mb2 = mb + a.n_groups;  // partner row block of a row-pair sweep
            const bool rows2 = kTwo && mb2 < a.n_mb;
            for (int vt = col; vt < a.n_vt && !aborted; vt += rows2 ? a.G : vstep) {
                const bool two = kTwo && (rows2 || vt + a.G < a.n_vt);
                // both CTAs' copies: H, the tile's W, and the partner block's H or the second tile's W
                const uint32_t stage_tx = 2u * (kStageBytesA + wb + (rows2 ? kStageBytesA : (two ? wb : 0u)));
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
                        ptx::tma_load_2d_pair(sB(stage, 0), &tmW, bar, w_x(kb),
                                              w_y(kb, vt * a.bn + (int)rank * half_bn), pol_w);
                        if (rows2)
                            ptx::tma_load_2d_pair(sB(stage, 1), &tmH, bar, kb * kBK,
                                                  mb2 * kPairM + (int)rank * kBM, pol_h);
                        else if (two)
                            ptx::tma_load_2d_pair(sB(stage, 1), &tmW, bar, w_x(kb),
                                                  w_y(kb, (vt + a.G) * a.bn + (int)rank * half_bn), pol_w);
                        if (tl && first)
                            tl[2] = ptx::globaltimer_ns();
                        first = false;
                    }
                    __syncwarp();
                    issued_parity[stage] = (int32_t)phase;
                    if (++stage == S) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
        }
        if (aborted && leader && lane == 0) {
            // Let every copy already issued (by either CTA) land before the pair's shared memory goes away.
            for (int s = 0; s < S; ++s)
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
            int item = 0;  // items issued so far
            bool aborted = false;
            auto wait_acc_free = [&](int i, uint32_t uses) -> bool {  // the epilogue has read use uses-1 of acc i
                int ok = 1;
                if (lane == 0)
                    ok = wait_bounded<true>(tempty(i), (uses & 1u) ^ 1u, &bars->abort);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                ptx::tc_fence_after();
                return ok != 0;
            };
            auto issue = [&](int acc, uint32_t a_smem, uint32_t b_smem, int kb) {  // 4 x K16 from one stage
                const uint64_t da = ptx::sdesc_kmajor_sw128(a_smem);
                const uint64_t db = ptx::sdesc_kmajor_sw128(b_smem);
#pragma unroll
                for (int k = 0; k < kBK / 16; ++k)  // +32 B along K per MMA = +2 in the encoded address
                    ptx::mma_bf16_pair(tmem + (uint32_t)acc * kBN, da + 2u * k, db + 2u * k, idesc, (kb | k) != 0);
            };
            for (int mb = grp; mb < a.n_mb && !aborted; mb += mb_step) {
                const bool rows2 = kTwo && mb + a.n_groups < a.n_mb;
                // accumulator 1 of a pass: the partner block's H (third slot) x the tile's W, or this block's
                // H x the second tile's W (third slot)
                auto issue1 = [&](int s, int kb) {
                    if (rows2)
                        issue(1, sB(s, 1), sB(s, 0), kb);
                    else
                        issue(1, sA(s), sB(s, 1), kb);
                };
                for (int vt = col; vt < a.n_vt && !aborted; vt += rows2 ? a.G : vstep, ++item) {
                    const bool two = kTwo && (rows2 || vt + a.G < a.n_vt);
                    // single tiles: item i uses accumulator i & 1 for the (i >> 1)-th time;
                    // passes: item i uses both accumulators for the i-th time
                    const int acc0 = kTwo ? 0 : (item & 1);
                    const uint32_t uses0 = kTwo ? (uint32_t)item : (uint32_t)(item >> 1);
                    if (!wait_acc_free(acc0, uses0)) {
                        aborted = true;
                        break;
                    }
                    const int defer = two ? min(S, a.n_kb) : 0;  // stages whose second-accumulator MMAs wait
                    const int s0 = stage;
                    for (int kb = 0; kb < a.n_kb; ++kb) {
                        int ok = 1;
                        if (lane == 0)
                            ok = wait_bounded(full(stage), phase, &bars->abort);
                        ok = __shfl_sync(0xffffffffu, ok, 0);
                        if (!ok) {
                            aborted = true;
                            break;
                        }
                        ptx::tc_fence_after();
                        if (lane == 0)
                            issue(acc0, sA(stage), sB(stage, 0), kb);
                        if (kb < defer) {
                            if (kb == defer - 1) {  // the second accumulator is needed now
                                if (!wait_acc_free(1, (uint32_t)item)) {
                                    aborted = true;
                                    break;
                                }
                                if (lane == 0)
                                    for (int j = 0; j < defer; ++j) {
                                        const int sj = (s0 + j) % S;
                                        issue1(sj, j);
                                        ptx::mma_commit_pair_multicast(empty(sj), kBothCtas);
                                    }
                            }
                        } else if (lane == 0) {
                            if (two)
                                issue1(stage, kb);
                            ptx::mma_commit_pair_multicast(empty(stage), kBothCtas);
                        }
                        __syncwarp();
                        if (++stage == S) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                    if (aborted)
                        break;
                    if (lane == 0) {
                        ptx::mma_commit_pair_multicast(tfull(acc0), kBothCtas);
                        if (kTwo)  // the epilogue waits for both accumulators of every pass
                            ptx::mma_commit_pair_multicast(tfull(1), kBothCtas);
                    }
                    __syncwarp();
                    tiles += two ? 2 : 1;
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
        const uint32_t lanes = tmem + ((uint32_t)(q * 32) << 16);
        int item = 0;
        bool aborted = false;
        auto take = [&](int i, uint32_t uses) -> bool {  // wait for use `uses` of accumulator i
            int ok = 1;
            if (lane == 0)
                ok = wait_bounded(tfull(i), uses & 1u, &bars->abort);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            ptx::tc_fence_after();
            return ok != 0;
        };
        auto release = [&](int i) {  // accumulator i fully read by this warp: tell the leader's MMA warp
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0)
                ptx::mbar_arrive_cluster(ptx::mapa(tempty(i), 0));
        };
        const RowState r0{-INFINITY, 0.f, 0.f, 0.f, 0.f, -INFINITY, 0.f, 0.f, 0.f, 0.f, 0};
        for (int mb = grp; mb < a.n_mb && !aborted; mb += mb_step) {
            const int mb2 = mb + a.n_groups;
            const bool rows2 = kTwo && mb2 < a.n_mb;
            const int64_t in_block = (int)rank * kBM + q * 32 + lane;
            const int64_t row = (int64_t)mb * kPairM + in_block;
            const int64_t row2 = rows2 ? (int64_t)mb2 * kPairM + in_block : (int64_t)a.N;  // a.N: no row
            const int32_t tgt = (row < a.N) ? row_target(a.ts, row, a.V) : -1;
            const int32_t tgt2 = (row2 < a.N) ? row_target(a.ts, row2, a.V) : -1;
            RowState r = r0, r2 = r0;  // r2: the partner block's row in a row-pair sweep
            for (int vt = col; vt < a.n_vt; vt += rows2 ? a.G : vstep, ++item) {
                const int acc0 = kTwo ? 0 : (item & 1);
                const uint32_t uses0 = kTwo ? (uint32_t)item : (uint32_t)(item >> 1);
                if (!take(acc0, uses0)) {
                    aborted = true;
                    break;
                }
                fold_tile<kEntropy>(r, lanes + (uint32_t)acc0 * kBN, vt * a.bn, min(a.bn, a.V - vt * a.bn), tgt);
                release(acc0);
                if (kTwo) {
                    if (!take(1, (uint32_t)item)) {
                        aborted = true;
                        break;
                    }
                    const int vt1 = vt + a.G;
                    if (rows2)
                        fold_tile<kEntropy>(r2, lanes + kBN, vt * a.bn, min(a.bn, a.V - vt * a.bn), tgt2);
                    else if (vt1 < a.n_vt)
                        fold_tile<kEntropy>(r, lanes + kBN, vt1 * a.bn, min(a.bn, a.V - vt1 * a.bn), tgt);
                    release(1);
                }
            }
            if (aborted)
                break;
#pragma unroll
            for (int i = 0; i < 2; ++i) {  // the previous sweep's records, then this sweep's become pending
                if (pend_idx[i] >= 0) {
                    a.part[pend_idx[i]] = pend[i];
                    if (kEntropy)
                        a.part_u[pend_idx[i]] = pend_u[i];
                }
                const RowState &x = i ? r2 : r;
                pend[i] = make_float4(x.m, (x.s0 + x.s1) + (x.s2 + x.s3), __int_as_float(x.am), x.tlog);
                pend_u[i] = (x.u0 + x.u1) + (x.u2 + x.u3);
                const int64_t rr = i ? row2 : row;
                pend_idx[i] = rr < a.N ? rr * a.G + col : -1;
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
    ptx::cluster_arrive_release();
#pragma unroll
    for (int i = 0; i < 2; ++i)
        if (pend_idx[i] >= 0) {
            a.part[pend_idx[i]] = pend[i];
            if (kEntropy)
                a.part_u[pend_idx[i]] = pend_u[i];
        }
    if (threadIdx.x == 64) {
        // Warp 2 has passed griddepcontrol.wait, so the previous call's finish kernel, which clears the
        // status word, has completed: a failure recorded now belongs to this call.
        if (!tmem_ok)
            atomicExch(&a.status->current, (int32_t)WINO_ERR_UNSUPPORTED);
        else if (*reinterpret_cast<volatile int32_t *>(&bars->abort))
            atomicExch(&a.status->current, (int32_t)WINO_ERR_DEVICE_TIMEOUT);
    }
    ptx::cluster_wait_acquire();
    ptx::tc_fence_after();
    if (warp == 1)
        ptx::tmem_dealloc_pair(tmem, kTmemCols);
    if (tl && threadIdx.x == 0)
        tl[6] = ptx::globaltimer_ns();
}

}  // namespace

// Choose the mode, the tile width bn and the number of row-block groups.  One 256-row block is bound by the
// W stream from HBM: single tiles (the most bytes in flight).  More rows are tensor-bound: passes (fewer bytes
// delivered per MMA; row-pair sweeps where a group owns more than one row block).  Then: fewest vocabulary columns on the busiest pair plus a per-tile or
// per-pass overhead, the widest tile, fewest passes over W (more groups).  A width below kBN pays when the
// vocabulary then splits evenly over the pairs: V = 126464 on 76 pairs is 494 tiles of 256 (7 on the
// busiest pair, 6.5 on average) but 527 tiles of 240 (7 on 71 pairs).
#ifndef WINO_PASS_MIN_ROW_BLOCKS
#define WINO_PASS_MIN_ROW_BLOCKS 2  // compile-time tuning: fewest 256-row blocks that use passes
#endif
constexpr int32_t kPassMinRowBlocks = WINO_PASS_MIN_ROW_BLOCKS;

ScoreSchedule score_schedule(int32_t n_mb, int64_t V, int max_units, int32_t records_cap)
{
    constexpr int64_t kTileOverheadCols = 16;  // single tiles: H re-staged per tile, in columns
    constexpr int64_t kPassOverheadCols = 32;  // passes: the epilogue the next pass partly waits for
    const int32_t two = n_mb >= kPassMinRowBlocks ? 1 : 0;
    ScoreSchedule best{kBN, (int32_t)((V + kBN - 1) / kBN), 1, 1, two, 2, 0};
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
            const int64_t tiles = (n_vt + g - 1) / g;  // on the busiest pair, per row block
            const int64_t per_mb = two ? tiles * bn + ((tiles + 1) / 2) * kPassOverheadCols
                                       : tiles * (bn + kTileOverheadCols);
            const int64_t cost = (int64_t)((n_mb + groups - 1) / groups) * per_mb;
            if (best_cost < 0 || cost < best_cost) {
                best_cost = cost;
                best.bn = bn;
                best.n_vt = (int32_t)n_vt;
                best.n_groups = groups;
                best.G = (int32_t)g;
            }
        }
    }
    // A pass stage has a third slot: the second tile's W, or in a row-pair sweep (a group with more than
    // one row block) the partner block's H.
    const uint32_t wb = stage_bytes_w(best.bn);
    const bool row_pairs = two && n_mb > best.n_groups;
    best.stage_bytes = kStageBytesA + wb + (two ? (row_pairs && wb < kStageBytesA ? kStageBytesA : wb) : 0u);
    const uint32_t fit = kRingCapacity / best.stage_bytes;
    best.stages = (int32_t)(fit < (uint32_t)kMaxStages ? fit : (uint32_t)kMaxStages);
    return best;
}

namespace {

cudaLaunchConfig_t score_config(unsigned grid, uint32_t smem, cudaStream_t stream, cudaLaunchAttribute (&attr)[2])
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kScoreThreads);
    cfg.dynamicSmemBytes = smem;
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
        for (auto *k : {score_kernel<false, false>, score_kernel<false, true>, score_kernel<true, false>,
                        score_kernel<true, true>})
            if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kScoreSmemMax) !=
                cudaSuccess)
                return -1;
        cudaLaunchAttribute attr[2];
        // Any launch's shared memory exceeds half an SM's, so one CTA per SM whatever the ring size.
        cudaLaunchConfig_t cfg = score_config(2, kScoreSmemMax, nullptr, attr);
        cfg.numAttrs = 1;  // the cluster shape is what matters for the occupancy query
        int clusters = 0;
        if (cudaOccupancyMaxActiveClusters(&clusters, score_kernel<false, true>, &cfg) != cudaSuccess || clusters < 1)
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
    // The ring must hold what the producer stages: a pass's third slot takes an H box (16 KB) in a row-pair
    // sweep, which the launch has when a group owns more than one row block.
    const uint32_t wb = stage_bytes_w(a.bn);
    const uint32_t third = a.two ? (a.n_mb > a.n_groups && wb < kStageBytesA ? kStageBytesA : wb) : 0u;
    if (a.stages < 2 || a.stages > kMaxStages || a.stage_bytes < kStageBytesA + wb + third ||
        a.stage_bytes % 1024u != 0 || (uint64_t)a.stages * a.stage_bytes > kRingCapacity)
        return cudaErrorInvalidValue;
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = score_config((unsigned)(2 * a.n_groups * a.G),
                                          kSmemOverhead + (uint32_t)a.stages * a.stage_bytes, stream, attr);
    if (entropy)
        return a.two ? cudaLaunchKernelEx(&cfg, score_kernel<true, true>, tmH, tmW, a)
                     : cudaLaunchKernelEx(&cfg, score_kernel<true, false>, tmH, tmW, a);
    return a.two ? cudaLaunchKernelEx(&cfg, score_kernel<false, true>, tmH, tmW, a)
                 : cudaLaunchKernelEx(&cfg, score_kernel<false, false>, tmH, tmW, a);
}

}  // namespace wino
