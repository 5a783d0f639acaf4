// finish.cu -- the end of a WINO step (sm_103a): merge the score kernel's
// partial softmax records per row, then apply Eq. 4 to the token state.
//
// finish_kernel: one warp per row folds the row's G partial records (fixed
// lane order, then a butterfly, so results are bit-for-bit reproducible) into
//   argmax   = smallest vocabulary id among the maximal logits,
//   pmax     = max_v p_v = 1 / sum_v exp(l_v - m),
//   ptarget  = p_target = exp(l_t - m) / sum_v exp(l_v - m)    (0 without a target),
// the three statistics Eq. 2 and Eq. 3 use, and on request the entropy
//   H(p)     = -sum_v p_v log p_v = ln Z - sum_v exp(l_v - m) (l_v - m) / Z
// that WINO+'s deferral and sharpening terms use (Sec. 5.3, Eq. 6-7).  In a whole step (wino_step) every
// CTA then adds its merged rows to its sequences' tickets; the CTA that
// completes a sequence's 2*L_b rows applies Eq. 4 to that sequence, so merge
// and update need one launch.  Tickets are cleared by the score kernel of the
// same step.  The kernel is launched programmatically: its launch overlaps the
// score kernel and it waits (griddepcontrol.wait) for the score kernel's
// results before touching them; it lets the next call's kernels launch at once
// (they only read H and W before their own griddepcontrol.wait).  The last of
// its CTAs publishes the call's status (see StatusWords).
//
// draft_verify_kernel: Eq. 4 alone from caller-supplied statistics
// (wino_draft_verify), one CTA per sequence.
//
// Eq. 4, per sequence, reading the state before the step y^(k-1):
//   draft  (Eq. 2): y_l == MASK and pmax(block row l) > tau1      -> argmax(block row l)
//   verify (Eq. 3): y_l != MASK and p(y_l | shadow row l) < tau2  -> MASK
// and, if no masked position clears tau1 while the block still has a MASK,
// the masked position with the largest pmax (smallest position on ties) is
// drafted: the greedy rule of Eq. 1, which keeps at least one token coming per
// step.  With draft_m > 0 the drafting rule is naive parallel sampling
// instead (Sec. 3): the draft_m masked positions with the largest pmax
// (smallest position first on ties) are drafted, whatever tau1 says.  The
// rules touch disjoint positions (MASK vs not MASK), so the update
// is applied in place in one pass after a CTA-wide reduction.  With
// WINO_OPT_FREEZE_FINISHED a sequence whose block already has no MASK is left
// as it is (its own loop, Sec. 4.2.3, has ended).
#include "internal.h"
#include "ptx.cuh"

namespace wino {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kFinishRows = 8;  // rows (warps) per finish CTA; also the CTA size of the Eq. 4 kernels

// Fold (m2, s2, i2) into (m, s, i): the larger max wins, the smaller index on equal maxima.
__device__ __forceinline__ void combine(float &m, float &s, int32_t &i, float m2, float s2, int32_t i2)
{
    const float M = fmaxf(m, m2);
    const float a = (m == -INFINITY) ? 0.f : s * ptx::ex2((m - M) * kLog2e);
    const float b = (m2 == -INFINITY) ? 0.f : s2 * ptx::ex2((m2 - M) * kLog2e);
    if (m2 > m || (m2 == m && i2 < i))
        i = i2;
    m = M;
    s = a + b;
}

// As combine, also folding u = sum exp(l - m) (l - m) log2(e) (rescaled to the new max like s).
__device__ __forceinline__ void combine_u(float &m, float &s, float &u, int32_t &i, float m2, float s2, float u2,
                                          int32_t i2)
{
    const float M = fmaxf(m, m2);
    float a = 0.f, b = 0.f, ua = 0.f, ub = 0.f;
    if (m != -INFINITY) {
        const float al = ptx::ex2((m - M) * kLog2e);
        a = s * al;
        ua = al * fmaf((m - M) * kLog2e, s, u);
    }
    if (m2 != -INFINITY) {
        const float bl = ptx::ex2((m2 - M) * kLog2e);
        b = s2 * bl;
        ub = bl * fmaf((m2 - M) * kLog2e, s2, u2);
    }
    if (m2 > m || (m2 == m && i2 < i))
        i = i2;
    m = M;
    s = a + b;
    u = ua + ub;
}

// Block-wide reduction scratch for eq4_block.
struct Eq4Smem {
    int32_t i0[kFinishRows], i1[kFinishRows], i2[kFinishRows];
    float f0[kFinishRows];
    float conf[kMaxBlkLen];  // fixed-M drafting: pmax of each masked position, -inf elsewhere
};

// Eq. 4 on sequence s by the whole CTA (kFinishRows warps; thread t owns positions t, t + 256, ...),
// reading the statistics of the a-th sequence of the scored rows (a = s unless an active-sequence list
// chose the rows).  Every load is issued before any decision so the update costs about one memory round
// trip.  Statistics are read through L2: other CTAs of the same launch may have written them.
__device__ void eq4_block(int a, int s, int32_t *tokens, const int32_t *argmax, const float *pmax,
                          const float *ptarget, const wino_params &p, int32_t *counts, int8_t *flags, int32_t status,
                          Eq4Smem &sm)
{
    constexpr int kT = kFinishRows * 32;
    constexpr int kPer = kMaxBlkLen / kT;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (status != WINO_OK) {  // the scores of this step are invalid: leave the state alone
        if (tid < 3)
            counts[s * 3 + tid] = status;
        return;
    }
    const int L = p.blk_len;
    const int32_t mask = p.mask_id;
    const bool shadow = !(p.options & WINO_OPT_NO_SHADOW);  // WINO+ inference has no verification rows
    const bool compact = (p.options & WINO_OPT_COMPACT) != 0;  // one row per position
    int32_t *y = tokens + (int64_t)s * p.seq_len + p.blk_start;
    const int64_t rb = (int64_t)((shadow && !compact) ? 2 * a : a) * L;  // rows read for masked positions
    const int64_t rs = (int64_t)(compact ? a : 2 * a + 1) * L;         // rows read for decoded positions

    int32_t yv[kPer], av[kPer];
    float pm[kPer], pt[kPer];
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        const int l = tid + i * kT;
        if (l < L) {
            yv[i] = y[l];
            av[i] = __ldcg(argmax + rb + l);
            pm[i] = __ldcg(pmax + rb + l);
            pt[i] = shadow ? __ldcg(ptarget + rs + l) : 1.0f;  // 1.0 is never below tau2 <= 1: no re-mask
        }
    }
    // Pass 1: how many masked positions clear tau1, and the most confident masked position.
    int n_clear = 0, n_mask = 0;
    float best = -INFINITY;
    int best_l = INT32_MAX;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        const int l = tid + i * kT;
        if (l < L && yv[i] == mask) {
            ++n_mask;
            n_clear += (pm[i] > p.tau1);
            if (pm[i] > best) {  // l grows with i: the first maximum keeps the smallest position
                best = pm[i];
                best_l = l;
            }
        }
    }
    n_clear = __reduce_add_sync(0xffffffffu, n_clear);
    n_mask = __reduce_add_sync(0xffffffffu, n_mask);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float b2 = __shfl_xor_sync(0xffffffffu, best, off);
        const int l2 = __shfl_xor_sync(0xffffffffu, best_l, off);
        if (b2 > best || (b2 == best && l2 < best_l)) {
            best = b2;
            best_l = l2;
        }
    }
    if (lane == 0) {
        sm.i0[warp] = n_clear;
        sm.i1[warp] = n_mask;
        sm.i2[warp] = best_l;
        sm.f0[warp] = best;
    }
    __syncthreads();
    n_clear = n_mask = 0;
    best = -INFINITY;
    best_l = INT32_MAX;
#pragma unroll
    for (int w = 0; w < kFinishRows; ++w) {
        n_clear += sm.i0[w];
        n_mask += sm.i1[w];
        if (sm.f0[w] > best || (sm.f0[w] == best && sm.i2[w] < best_l)) {
            best = sm.f0[w];
            best_l = sm.i2[w];
        }
    }
    __syncthreads();  // the scratch is reused below
    if (n_mask == 0 && (p.options & WINO_OPT_FREEZE_FINISHED)) {  // finished block: its loop has stopped
        if (flags)
            for (int l = tid; l < L; l += kT)
                flags[(int64_t)s * L + l] = 0;
        if (tid < 3)
            counts[s * 3 + tid] = 0;
        return;
    }
    const int fallback = (p.draft_m <= 0 && n_clear == 0 && n_mask > 0) ? best_l : -1;

    // Fixed-M drafting: position l is drafted iff fewer than M masked positions rank before it
    // (larger pmax, or equal pmax and a smaller position).
    bool top[kPer];
#pragma unroll
    for (int i = 0; i < kPer; ++i)
        top[i] = false;
    if (p.draft_m > 0) {
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
            const int l = tid + i * kT;
            if (l < L)
                sm.conf[l] = (yv[i] == mask) ? pm[i] : -INFINITY;
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
            const int l = tid + i * kT;
            if (l < L && yv[i] == mask) {
                int before = 0;
                for (int j = 0; j < L && before < p.draft_m; ++j) {
                    const float c = sm.conf[j];
                    before += (c > pm[i]) || (c == pm[i] && j < l);
                }
                top[i] = before < p.draft_m;
            }
        }
        __syncthreads();  // conf is scratch of this sequence only
    }

    // Pass 2: apply Eq. 4 simultaneously.
    int drafted = 0, remasked = 0, left = 0;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        const int l = tid + i * kT;
        if (l >= L)
            break;
        const int32_t prev = yv[i];
        int32_t next = prev;
        int8_t code = 0;
        if (prev == mask) {
            if (p.draft_m > 0 ? top[i] : (pm[i] > p.tau1 || l == fallback)) {
                next = av[i];
                code = (next == mask) ? 4 : (p.draft_m > 0 ? 5 : (l == fallback ? 2 : 1));
            }
        } else if (shadow && pt[i] < p.tau2) {
            next = mask;
            code = 3;
        }
        if (next != prev) {
            y[l] = next;
            if (p.last_change)  // WINO finalization step bookkeeping (Sec. 5.1)
                p.last_change[(int64_t)s * p.seq_len + p.blk_start + l] = p.step_index;
        }
        drafted += (code == 1 || code == 2 || code == 5);
        remasked += (code == 3);
        left += (next == mask);
        if (flags)
            flags[(int64_t)s * L + l] = code;
    }
    drafted = __reduce_add_sync(0xffffffffu, drafted);
    remasked = __reduce_add_sync(0xffffffffu, remasked);
    left = __reduce_add_sync(0xffffffffu, left);
    if (lane == 0) {
        sm.i0[warp] = drafted;
        sm.i1[warp] = remasked;
        sm.i2[warp] = left;
    }
    __syncthreads();
    if (tid < 3) {
        const int32_t *src = tid == 0 ? sm.i0 : (tid == 1 ? sm.i1 : sm.i2);
        int32_t v = 0;
#pragma unroll
        for (int w = 0; w < kFinishRows; ++w)
            v += src[w];
        counts[s * 3 + tid] = v;
    }
    __syncthreads();  // the scratch may be reused for the next sequence
}

// Eq. 4: the CTA that merges the last rows of a sequence updates that sequence.
__device__ void eq4_tail(const FinishArgs &a, int64_t row0, int32_t status, int32_t *s_done, int32_t &s_ndone,
                         Eq4Smem &sm)
{
    __syncthreads();
    if (threadIdx.x == 0) {
        int32_t nd = 0;
        const int64_t per_seq =
            ((a.p.options & (WINO_OPT_NO_SHADOW | WINO_OPT_COMPACT)) ? 1 : 2) * (int64_t)a.p.blk_len;
        const int64_t rend = min(row0 + kFinishRows, (int64_t)a.N);
        for (int64_t r = row0; r < rend;) {
            const int64_t sq = r / per_seq;
            const int64_t send = min((sq + 1) * per_seq, rend);
            const int32_t cnt = (int32_t)(send - r);
            if (atomicAdd(&a.tickets[sq], cnt) + cnt == per_seq)
                s_done[nd++] = (int32_t)sq;
            r = send;
        }
        s_ndone = nd;
        __threadfence();
    }
    __syncthreads();
    const int nd = s_ndone;
    for (int i = 0; i < nd; ++i) {
        const int sq = a.p.active_seq ? a.p.active_seq[s_done[i]] : s_done[i];
        if (sq < 0 || sq >= a.p.n_seq) {  // a bad entry of the caller's list: no update, an error status
            if (threadIdx.x == 0)
                atomicExch(&a.status->current, (int32_t)WINO_ERR_ARG);
            continue;
        }
        eq4_block(s_done[i], sq, a.tokens, a.argmax, a.pmax, a.ptarget, a.p, a.counts, a.flags, status, sm);
    }
}

__global__ void __launch_bounds__(kFinishRows * 32) finish_kernel(const FinishArgs a)
{
    ptx::grid_dep_launch_dependents();  // the next call may start streaming its H and W
    ptx::grid_dep_wait();
    __shared__ int32_t s_done[kFinishRows];
    __shared__ int32_t s_ndone;
    __shared__ Eq4Smem sm;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t row0 = (int64_t)blockIdx.x * kFinishRows;
    const int64_t row = row0 + warp;
    const int32_t status = *reinterpret_cast<volatile int32_t *>(&a.status->current);

    if (row < a.N) {
        if (status != WINO_OK) {
            if (lane == 0) {
                a.argmax[row] = -1;
                a.pmax[row] = __int_as_float(0x7fc00000);
                a.ptarget[row] = __int_as_float(0x7fc00000);
                if (a.entropy)
                    a.entropy[row] = __int_as_float(0x7fc00000);
            }
        } else {
            const float4 *pr = a.part + row * a.G;
            // every record of the row (G <= 8 * 32) and the target's record are loaded at once
            constexpr int kRec = kMaxRecordsPerRow / 32;
            float4 r[kRec];
#pragma unroll
            for (int i = 0; i < kRec; ++i) {
                const int j = lane + 32 * i;
                r[i] = (j < a.G) ? __ldcg(pr + j) : make_float4(-INFINITY, 0.f, __int_as_float(INT32_MAX), -INFINITY);
            }
            // The record of the pair whose tiles hold the row's target carries its logit; the others -inf.
            float m = -INFINITY, s = 0.f, tl = -INFINITY, u = 0.f;
            int32_t idx = INT32_MAX;
            if (!a.entropy) {
#pragma unroll
                for (int i = 0; i < kRec; ++i) {
                    combine(m, s, idx, r[i].x, r[i].y, __float_as_int(r[i].z));
                    tl = fmaxf(tl, r[i].w);
                }
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) {
                    const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
                    const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
                    const int32_t i2 = __shfl_xor_sync(0xffffffffu, idx, off);
                    tl = fmaxf(tl, __shfl_xor_sync(0xffffffffu, tl, off));
                    combine(m, s, idx, m2, s2, i2);
                }
            } else {
                const float *pu = a.part_u + row * a.G;
#pragma unroll
                for (int i = 0; i < kRec; ++i) {
                    const int j = lane + 32 * i;
                    combine_u(m, s, u, idx, r[i].x, r[i].y, (j < a.G) ? __ldcg(pu + j) : 0.f,
                              __float_as_int(r[i].z));
                    tl = fmaxf(tl, r[i].w);
                }
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) {
                    const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
                    const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
                    const float u2 = __shfl_xor_sync(0xffffffffu, u, off);
                    const int32_t i2 = __shfl_xor_sync(0xffffffffu, idx, off);
                    tl = fmaxf(tl, __shfl_xor_sync(0xffffffffu, tl, off));
                    combine_u(m, s, u, idx, m2, s2, u2, i2);
                }
            }
            if (lane == 0) {
                a.argmax[row] = idx;
                a.pmax[row] = 1.0f / s;
                a.ptarget[row] = (tl > -INFINITY) ? ptx::ex2((tl - m) * kLog2e) / s : 0.0f;
                if (a.entropy)  // H = ln Z - (u ln 2) / Z, with u in log2 units
                    a.entropy[row] = (ptx::lg2(s) - u / s) * kLn2;
                __threadfence();  // publish this row before the CTA signals its ticket
            }
        }
    }
    if (a.tokens)
        eq4_tail(a, row0, status, s_done, s_ndone, sm);

    // The last CTA done with this call publishes its status and clears the word for the next call.
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        if (atomicAdd(&a.status->finished, 1u) == gridDim.x - 1) {
            __threadfence();
            a.status->last = atomicExch(&a.status->current, (int32_t)WINO_OK);
        }
    }
}

// Eq. 4 alone, one CTA per sequence.
__global__ void __launch_bounds__(kFinishRows * 32)
    draft_verify_kernel(int32_t *tokens, const int32_t *argmax, const float *pmax, const float *ptarget,
                        const wino_params p, int32_t *counts, int8_t *flags)
{
    __shared__ Eq4Smem sm;
    eq4_block(blockIdx.x, blockIdx.x, tokens, argmax, pmax, ptarget, p, counts, flags, WINO_OK, sm);
}

// Row compaction: one CTA per position copies the one row Eq. 4 will read -- the block row of a masked
// position, the shadow row of a decoded one -- with 16-byte loads (d % 8 == 0).
__global__ void __launch_bounds__(256) gather_compact_kernel(const uint4 *__restrict__ H, uint4 *__restrict__ Hc,
                                                             const int32_t *__restrict__ tokens, const wino_params p,
                                                             int64_t vec_per_row)
{
    ptx::grid_dep_launch_dependents();  // the score kernel may set up now; it waits for these rows itself
    ptx::grid_dep_wait();  // the token state may still be being written by the previous step
    const int64_t r = blockIdx.x;  // = s * L + l
    const int64_t s = r / p.blk_len, l = r - s * p.blk_len;
    const bool masked = tokens[s * p.seq_len + p.blk_start + l] == p.mask_id;
    const uint4 *src = H + ((2 * s + (masked ? 0 : 1)) * p.blk_len + l) * vec_per_row;
    uint4 *dst = Hc + r * vec_per_row;
    for (int64_t i = threadIdx.x; i < vec_per_row; i += blockDim.x)
        dst[i] = __ldg(src + i);
}

// Active-sequence gather: one CTA per scored row copies the row of a listed sequence (row r of the
// gathered layout belongs to the a-th listed sequence s) into the workspace with 16-byte loads, and
// writes the row's target: the current token of the position a shadow row verifies, else -1 (MASK or
// a block row), so that the score kernel reads the gathered rows with explicit targets.
__global__ void __launch_bounds__(256) gather_active_kernel(const uint4 *__restrict__ H, uint4 *__restrict__ Hc,
                                                            int32_t *__restrict__ target,
                                                            const int32_t *__restrict__ tokens, const wino_params p,
                                                            int64_t vec_per_row)
{
    ptx::grid_dep_launch_dependents();  // the score kernel waits for these rows itself
    ptx::grid_dep_wait();  // the token state may still be being written by the previous step
    const bool shadow = !(p.options & WINO_OPT_NO_SHADOW);
    const bool compact = (p.options & WINO_OPT_COMPACT) != 0;
    const int64_t L = p.blk_len;
    const int64_t per_seq = (shadow && !compact) ? 2 * L : L;
    const int64_t r = blockIdx.x;
    const int64_t a = r / per_seq, j = r - a * per_seq;
    const int64_t s = p.active_seq[a];
    uint4 *dst = Hc + r * vec_per_row;
    if (s < 0 || s >= p.n_seq) {  // a bad entry of the caller's list: read nothing (the finish kernel reports it)
        for (int64_t i = threadIdx.x; i < vec_per_row; i += blockDim.x)
            dst[i] = make_uint4(0, 0, 0, 0);
        if (threadIdx.x == 0)
            target[r] = -1;
        return;
    }
    const int64_t l = (j < L) ? j : j - L;
    const int32_t y = tokens[s * p.seq_len + p.blk_start + l];
    // kind of the row: the shadow row for j >= L; with compaction, the row Eq. 4 reads for this position
    const int kind = !shadow ? 0 : (compact ? (y == p.mask_id ? 0 : 1) : (j < L ? 0 : 1));
    const int64_t src_row = shadow ? (2 * s + kind) * L + l : s * L + l;
    const uint4 *src = H + src_row * vec_per_row;
    for (int64_t i = threadIdx.x; i < vec_per_row; i += blockDim.x)
        dst[i] = __ldg(src + i);
    if (threadIdx.x == 0)
        target[r] = (kind == 1 && y != p.mask_id) ? y : -1;
}

}  // namespace

cudaError_t launch_gather_compact(const uint16_t *H, uint16_t *Hc, const int32_t *tokens, const wino_params &p,
                                  int64_t d, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((int64_t)p.n_seq * p.blk_len));
    cfg.blockDim = dim3(256);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, gather_compact_kernel, reinterpret_cast<const uint4 *>(H),
                              reinterpret_cast<uint4 *>(Hc), tokens, p, d / 8);
}

cudaError_t launch_gather_active(const uint16_t *H, uint16_t *Hc, int32_t *target, const int32_t *tokens,
                                 const wino_params &p, int64_t rows, int64_t d, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)rows);
    cfg.blockDim = dim3(256);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, gather_active_kernel, reinterpret_cast<const uint4 *>(H),
                              reinterpret_cast<uint4 *>(Hc), target, tokens, p, d / 8);
}

cudaError_t launch_finish(const FinishArgs &a, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((a.N + kFinishRows - 1) / kFinishRows));
    cfg.blockDim = dim3(kFinishRows * 32);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, finish_kernel, a);
}

cudaError_t launch_draft_verify(int32_t *tokens, const int32_t *argmax, const float *pmax, const float *ptarget,
                                const wino_params &p, int32_t *counts, int8_t *flags, cudaStream_t stream)
{
    draft_verify_kernel<<<p.n_seq, kFinishRows * 32, 0, stream>>>(tokens, argmax, pmax, ptarget, p, counts, flags);
    return cudaGetLastError();
}

}  // namespace wino
