// draft_verify.cu -- the WINO update of the token state, Eq. 4 (sm_103a).
//
// One warp per sequence; lane j owns block positions j, j + 32, ...  Both
// rules read the state before the step, y^(k-1):
//   draft  (Eq. 2): y_l == MASK and pmax(block row l) > tau1   -> argmax(block row l)
//   verify (Eq. 3): y_l != MASK and p(y_l | shadow row l) < tau2 -> MASK
// and if no masked position clears tau1 while the block still has a MASK,
// the masked position with the largest pmax (smallest position on ties) is
// drafted: the greedy rule of Eq. 1, which keeps at least one token coming
// per step.  The two rules touch disjoint positions (MASK vs not MASK), so
// the update is applied in place in one pass after a warp-wide reduction.
#include "internal.h"

namespace wino {
namespace {

constexpr int kWarpsPerBlock = 4;

__global__ void __launch_bounds__(kWarpsPerBlock * 32)
    draft_verify_kernel(int32_t *__restrict__ tokens, const int32_t *__restrict__ argmax,
                        const float *__restrict__ pmax, const float *__restrict__ ptarget, const wino_params p,
                        int32_t *__restrict__ counts, int8_t *__restrict__ flags, const int32_t *__restrict__ status)
{
    const int s = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (s >= p.n_seq)
        return;
    if (status && *status != WINO_OK) {  // the scores of this step are invalid: leave the state alone
        if (lane < 3)
            counts[s * 3 + lane] = *status;
        return;
    }
    const int L = p.blk_len;
    const int32_t mask = p.mask_id;
    int32_t *y = tokens + (int64_t)s * p.seq_len + p.blk_start;
    const int64_t rb = (int64_t)(2 * s) * L;      // kind-0 rows: the block Y_cur
    const int64_t rs = (int64_t)(2 * s + 1) * L;  // kind-1 rows: the shadow block Y_shad

    // Pass 1: how many masked positions clear tau1, and the most confident masked position.
    int n_clear = 0, n_mask = 0;
    float best = -INFINITY;
    int best_l = INT32_MAX;
    for (int l = lane; l < L; l += 32) {
        if (y[l] == mask) {
            const float pm = pmax[rb + l];
            ++n_mask;
            n_clear += (pm > p.tau1);
            if (pm > best || (pm == best && l < best_l)) {
                best = pm;
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
    const int fallback = (n_clear == 0 && n_mask > 0) ? best_l : -1;

    // Pass 2: apply Eq. 4 simultaneously.
    int drafted = 0, remasked = 0, left = 0;
    for (int l = lane; l < L; l += 32) {
        const int32_t prev = y[l];
        int32_t next = prev;
        int8_t code = 0;
        if (prev == mask) {
            if (pmax[rb + l] > p.tau1 || l == fallback) {
                next = argmax[rb + l];
                code = (next == mask) ? 4 : (l == fallback ? 2 : 1);
            }
        } else if (ptarget[rs + l] < p.tau2) {
            next = mask;
            code = 3;
        }
        if (next != prev)
            y[l] = next;
        drafted += (code == 1 || code == 2);
        remasked += (code == 3);
        left += (next == mask);
        if (flags)
            flags[(int64_t)s * L + l] = code;
    }
    drafted = __reduce_add_sync(0xffffffffu, drafted);
    remasked = __reduce_add_sync(0xffffffffu, remasked);
    left = __reduce_add_sync(0xffffffffu, left);
    if (lane == 0) {
        counts[s * 3 + 0] = drafted;
        counts[s * 3 + 1] = remasked;
        counts[s * 3 + 2] = left;
    }
}

}  // namespace

cudaError_t launch_draft_verify(int32_t *tokens, const int32_t *argmax, const float *pmax, const float *ptarget,
                                const wino_params &p, int32_t *counts, int8_t *flags, const int32_t *status,
                                cudaStream_t stream)
{
    const int blocks = (p.n_seq + kWarpsPerBlock - 1) / kWarpsPerBlock;
    draft_verify_kernel<<<blocks, kWarpsPerBlock * 32, 0, stream>>>(tokens, argmax, pmax, ptarget, p, counts, flags,
                                                                     status);
    return cudaGetLastError();
}

}  // namespace wino
