// internal.h -- declarations shared by the translation units of libwino.so (not installed).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "wino.h"

namespace wino {

// Scoring tile: a CTA pair (2-SM tcgen05 MMA, cta_group::2) computes 256 rows
// of H x bn vocabulary columns (bn <= 256, a multiple of 16, chosen per launch
// by score_schedule so that the vocabulary splits evenly over the pairs).  Per
// 64-wide K slice each CTA stages its own 128 rows of H and bn/2 of the tile's
// bn W rows (128-byte swizzle rows) in a ring of shared-memory stages, and
// holds its 128 rows x bn columns of the fp32 accumulator in TMEM (one TMEM
// lane per row).  Two fp32 accumulators fill TMEM's 512 columns; a launch uses
// them in one of two modes (ScoreArgs::two):
//   single tiles: the accumulators alternate, so the epilogue of one tile
//     overlaps the MMAs of the next; stages of 16 KB + bn*64 B, up to 7 of them
//     (the most bytes in flight, for shapes bound by the W stream from HBM);
//   passes (tensor-bound shapes): a stage holds three slots multiplied into
//     both accumulators, a quarter fewer bytes delivered per SM and MMA.  Two
//     row blocks of a group share each W slice (row-pair sweep: H, W, H), so
//     the group reads W from HBM once per two blocks; a block without a partner
//     shares its H slice between two tiles (tile-pair sweep: H, W, W).
constexpr int kPairM = 256;  // rows per pair tile (UMMA M)
constexpr int kBM = 128;     // rows per CTA
constexpr int kBN = 256;     // largest tile width (UMMA N); TMEM column stride of the two accumulators
constexpr int kMinBN = 128;  // narrowest tile width the schedule uses
constexpr int kBK = 64;
constexpr int kMaxStages = 7;
constexpr int kScoreThreads = 192;  // warp 0 TMA, warp 1 TMEM + MMA, warps 2-5 epilogue
constexpr uint32_t kStageBytesA = kBM * kBK * 2;  // 16 KB of H per stage
constexpr uint32_t kScoreSmemMax = 227u * 1024u;  // the most dynamic shared memory a CTA may have
constexpr uint32_t kSmemOverhead = 1024 /* ring alignment slack */ + 256 /* barriers */;
constexpr uint32_t kRingCapacity = kScoreSmemMax - kSmemOverhead;
constexpr uint32_t kTmemCols = 2 * kBN;  // two 256-column fp32 accumulators: all 512 TMEM columns

// W bytes one CTA stages per K slice of a tile of width bn (bn/2 rows of 128 B; a multiple of 1 KB).
__host__ __device__ constexpr uint32_t stage_bytes_w(int bn) { return (uint32_t)(bn / 2) * kBK * 2; }

constexpr int kMaxBlkLen = 1024;

// Where a scored row's target token comes from.
struct TargetSource {
    const int32_t *target;  // explicit per-row targets (wino_score_rows), or nullptr
    const int32_t *tokens;  // or gathered from the token state (wino_step), or nullptr
    int32_t seq_len, blk_start, blk_len, mask_id;
    int32_t compact;        // rows are one per position (s, l) -> row s*blk_len + l (WINO_OPT_COMPACT)
};

// Target of row `row`: explicit, or the current token of the position a
// shadow (kind-1) row verifies; -1 when there is none or it is outside [0, V).
__device__ __forceinline__ int32_t row_target(const TargetSource &ts, int64_t row, int32_t V)
{
    int32_t t = -1;
    if (ts.target) {
        t = ts.target[row];
    } else if (ts.tokens && ts.compact) {
        // one row per position: a decoded position's row is its shadow row, scored against its token
        const int64_t s = row / ts.blk_len, l = row - s * ts.blk_len;
        const int32_t y = ts.tokens[s * ts.seq_len + ts.blk_start + l];
        t = (y == ts.mask_id) ? -1 : y;
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

// Work split of the score kernel.  The 256-row blocks are spread over n_groups
// groups of G CTA pairs; pair c serves row blocks c % n_groups (+ n_groups, ...)
// and, within each, vocabulary tiles c / n_groups (+ G, ...).  The G pairs of a
// group walk the vocabulary side by side, so all groups read the same W tiles
// at the same time (W streams from HBM once per sweep), and each CTA keeps its
// running softmax state per row across its tiles and writes ONE partial record
// per (row, pair of the group): G records per row.
constexpr int kMaxRecordsPerRow = 256;

// Status words at the start of every workspace.  `current` collects the
// errors of the call in flight: score-kernel CTAs record theirs only after
// griddepcontrol.wait (so after the previous call's finish kernel has cleared
// the word), and the finish kernel adds its own.  The last finish CTA of a call
// publishes `current` as `last` (what wino_read_device_status returns) and
// clears it for the next call; `finished` counts the finish CTAs done with the
// call and is reset by the next call's score kernel.  A workspace starts zeroed.
struct StatusWords {
    int32_t current;
    int32_t last;
    uint32_t finished;
};

// Optional per-CTA timeline of the score kernel (diagnostics, off by default):
// kTimelineWords 64-bit words per CTA, see score.cu.
constexpr int kTimelineWords = 8;

// Partial record: running max logit m, sum of exp(l - m), argmax (int bits),
// logit of the row's target if the target lies in one of the pair's tiles (else -inf).
struct ScoreArgs {
    int32_t N, d, V;
    int32_t n_mb, n_vt, n_kb;  // n_mb: 256-row blocks, n_vt: vocabulary tiles of bn columns
    int32_t bn;                // tile width (multiple of 16, kMinBN..kBN)
    int32_t two;               // 1: passes, 0: single tiles (see above)
    int32_t stages;            // ring stages, 2..kMaxStages
    uint32_t stage_bytes;      // 16 KB + stage_bytes_w(bn) + a pass's third slot (W, or 16 KB of H)
    int32_t n_groups, G;
    TargetSource ts;
    float4 *part;       // [N][G]
    float *part_u;      // [N][G], entropy variant only: sum of exp(l - m) * (l - m) * log2(e) over the pair's tiles
    StatusWords *status;
    int32_t *tickets;   // [n_tickets], cleared here for the finish kernel
    int32_t n_tickets;
    uint64_t *timeline;        // nullptr, or [gridDim.x][kTimelineWords] stamps of this launch
    int32_t w_panels;          // W's tensor map is over the panel copy [d/64 * V, 64]: row v of K slice kb at kb * V + v
};

struct FinishArgs {
    const float4 *part;
    const float *part_u;  // with entropy != nullptr
    float *entropy;       // optional: H(p) = -sum_v p_v log p_v per row
    int32_t G, N, V;
    TargetSource ts;
    StatusWords *status;  // read; WINO_ERR_ARG added when an active-sequence list entry is out of range
    int32_t *argmax;
    float *pmax;
    float *ptarget;
    // Eq. 4 in the same launch when tokens != nullptr (wino_step)
    int32_t *tokens;
    wino_params p;
    int32_t *counts;
    int8_t *flags;
    int32_t *tickets;  // [n_seq], zero on entry
};

// Work split of one score launch: tile width bn, number of row-block groups and pairs per group, for
// n_mb 256-row blocks over a vocabulary of V entries on max_units resident pairs.  At most
// records_cap records per row (the workspace holds that many).
struct ScoreSchedule {
    int32_t bn, n_vt, n_groups, G;
    int32_t two, stages;
    uint32_t stage_bytes;
};
ScoreSchedule score_schedule(int32_t n_mb, int64_t V, int max_units, int32_t records_cap);

// Records per row the workspace reserves for a vocabulary of V entries: one per tile at the narrowest
// width, at most kMaxRecordsPerRow.
inline int64_t records_per_row(int64_t V)
{
    const int64_t n = (V + kMinBN - 1) / kMinBN;
    return n < kMaxRecordsPerRow ? n : kMaxRecordsPerRow;
}

// CTA pairs of the score kernel that can be resident at once on the current device (<= 0 on error).
int score_max_pairs();

// entropy: also accumulate part_u (the variant used when wino_score_rows is asked for H(p)).
cudaError_t launch_score(const CUtensorMap &tmH, const CUtensorMap &tmW, const ScoreArgs &a, bool entropy,
                         cudaStream_t stream);

cudaError_t launch_finish(const FinishArgs &a, cudaStream_t stream);

// Row compaction (WINO_OPT_COMPACT): Hc[s*L + l] = H[(2s + (tokens[s, b0 + l] == MASK ? 0 : 1)) * L + l].
cudaError_t launch_gather_active(const uint16_t *H, uint16_t *Hc, int32_t *target, const int32_t *tokens,
                                 const wino_params &p, int64_t rows, int64_t d, cudaStream_t stream);
cudaError_t launch_gather_compact(const uint16_t *H, uint16_t *Hc, const int32_t *tokens, const wino_params &p,
                                  int64_t d, cudaStream_t stream);

// Wp[k][v][c] = W[v][64k + c] (wino_lm_head_panels); d a multiple of 64, (d/64) * V <= 2^30.
cudaError_t launch_panels(const uint16_t *W, uint16_t *Wp, int64_t d, int64_t V, int sm_count, cudaStream_t stream);

cudaError_t launch_draft_verify(int32_t *tokens, const int32_t *argmax, const float *pmax, const float *ptarget,
                                const wino_params &p, int32_t *counts, int8_t *flags, cudaStream_t stream);

}  // namespace wino
