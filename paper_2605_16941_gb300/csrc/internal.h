// internal.h -- declarations shared by the translation units of libwino.so (not installed).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "wino.h"

namespace wino {

// Scoring tile: 128 rows of H (one TMEM lane each) x 256 vocabulary columns
// (the UMMA N extent and one 256-column TMEM accumulator), K staged 64 bf16
// (one 128-byte swizzle row) at a time through a 4-deep shared-memory ring.
constexpr int kBM = 128;
constexpr int kBN = 256;
constexpr int kBK = 64;
constexpr int kStages = 4;
constexpr int kScoreThreads = 192;  // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr uint32_t kStageBytesA = kBM * kBK * 2;  // 16 KB
constexpr uint32_t kStageBytesB = kBN * kBK * 2;  // 32 KB
constexpr uint32_t kRingBytes = kStages * (kStageBytesA + kStageBytesB);
constexpr uint32_t kScoreSmemBytes = kRingBytes + 1024 /* alignment slack */ + 256 /* barriers */;
constexpr uint32_t kTmemCols = 2 * kBN;  // double-buffered fp32 accumulator

constexpr int kMaxBlkLen = 1024;

// Where a scored row's target token comes from.
struct TargetSource {
    const int32_t *target;  // explicit per-row targets (wino_score_rows), or nullptr
    const int32_t *tokens;  // or gathered from the token state (wino_step), or nullptr
    int32_t seq_len, blk_start, blk_len, mask_id;
};

// Target of row `row`: explicit, or the current token of the position a
// shadow (kind-1) row verifies; -1 when there is none or it is outside [0, V).
__device__ __forceinline__ int32_t row_target(const TargetSource &ts, int64_t row, int32_t V)
{
    int32_t t = -1;
    if (ts.target) {
        t = ts.target[row];
    } else if (ts.tokens) {
        const int64_t two_l = 2 * (int64_t)ts.blk_len;
        const int64_t s = row / two_l, r = row - s * two_l;
        if (r >= ts.blk_len) {
            const int32_t y = ts.tokens[s * ts.seq_len + ts.blk_start + (r - ts.blk_len)];
            t = (y == ts.mask_id) ? -1 : y;
        }
    }
    return (t >= 0 && t < V) ? t : -1;
}

// One partial softmax record per (row, vocabulary tile): running max logit m,
// sum of exp(l - m) over the tile, argmax (int bits) and the target's logit
// when the target lies in the tile (else 0).  Layout [row][tile].
struct ScoreArgs {
    int32_t N, d, V;
    int32_t n_mb, n_vt, n_kb;
    int64_t n_tiles;
    TargetSource ts;
    float4 *part;
    int32_t *status;
};

cudaError_t launch_score(const CUtensorMap &tmH, const CUtensorMap &tmW, const ScoreArgs &a, int grid,
                         cudaStream_t stream);

cudaError_t launch_merge(const float4 *part, int32_t N, int32_t n_vt, int32_t V, const TargetSource &ts,
                         const int32_t *status, int32_t *argmax, float *pmax, float *ptarget, cudaStream_t stream);

cudaError_t launch_draft_verify(int32_t *tokens, const int32_t *argmax, const float *pmax, const float *ptarget,
                                const wino_params &p, int32_t *counts, int8_t *flags, const int32_t *status,
                                cudaStream_t stream);

}  // namespace wino
