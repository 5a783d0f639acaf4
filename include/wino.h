/*
 * wino.h -- C ABI of the GB300 (sm_103a) WINO scoring-and-revoke step.
 *
 * WINO ("Wide-In, Narrow-Out", arXiv 2605.16941, Sec. 4) decodes a block of a
 * diffusion LLM's response by drafting and verifying in one forward pass.
 * Per step and per sequence it scores 2*L_b rows of hidden states through
 * the LM head: L_b rows of the current block Y_cur (drafting, Eq. 2) and L_b
 * rows of the shadow block Y_shad (verification, Eq. 3), then applies Eq. 4:
 *   - a masked position whose block row has max_v p > tau1 takes that row's
 *     argmax token (Eq. 2); if no masked position clears tau1, the single
 *     most confident masked position is drafted anyway (greedy rule, Eq. 1);
 *   - a decoded position whose shadow row gives its current token a
 *     probability < tau2 is re-masked (Eq. 3);
 *   - everything else, and every position outside the block, is unchanged.
 *
 * Conventions shared by every entry point
 *   - Every array argument is a DEVICE pointer owned by the caller unless
 *     marked host; the library never allocates, frees or synchronises
 *     (except wino_read_device_status, which reads back one word, and
 *     wino_decode, whose loop reads each step's counts back).
 *   - bf16 data are passed as uint16_t bit patterns (IEEE binary32 top half).
 *   - Alignment: H and W 16 bytes, workspaces 256 bytes, int32 and float
 *     arrays 4 bytes; a misaligned pointer is rejected with WINO_ERR_ARG
 *     before anything is launched.
 *   - Row order of the scored rows is [s][kind][l]: sequence s, kind 0 = the
 *     current-block row of position l, kind 1 = its shadow-block row; row
 *     index n = (2*s + kind)*blk_len + l, N = 2*n_seq*blk_len.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream); all work is
 *     enqueued on it asynchronously, in order.  The kernels are launched with
 *     programmatic dependent launch: a call's first kernel sets up (barriers,
 *     tensor memory, L2 prefetches of its first H and W tiles) while the
 *     kernel before it on the stream finishes, and reads nothing from global
 *     memory until that kernel has completed, whatever it is.
 *   - Return value: WINO_OK (0) or a negative wino_status.  On an argument
 *     error nothing is enqueued.  Device-side failures (a bounded wait that
 *     expired) are reported through the workspace's status words, see
 *     wino_read_device_status.
 *   - Devices: compute capability 10.3 (GB300).  Other devices get
 *     WINO_ERR_UNSUPPORTED.
 */
#ifndef WINO_H
#define WINO_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define WINO_API __attribute__((visibility("default")))
#else
#define WINO_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    WINO_OK = 0,
    WINO_ERR_ARG = -1,            /* null pointer, misaligned pointer, threshold out of range  */
    WINO_ERR_SHAPE = -2,          /* sizes outside the supported range (see each call)         */
    WINO_ERR_WORKSPACE = -3,      /* ws_bytes below wino_workspace_size(), or a problem larger
                                     than the fixed array of wino_step_static_scratch          */
    WINO_ERR_CUDA = -4,           /* a CUDA runtime/driver call or kernel launch failed        */
    WINO_ERR_MAX_STEPS = -5,      /* a decode loop exceeded its step budget (loop drivers)     */
    WINO_ERR_DEVICE_TIMEOUT = -6, /* a bounded device-side wait expired; outputs are invalid   */
    WINO_ERR_UNSUPPORTED = -7     /* not a compute-capability 10.3 device                      */
} wino_status;

/* Decoding parameters (host memory, read during the call only). */
typedef struct {
    float tau1;        /* drafting threshold, Eq. 2: draft iff max_v p > tau1 (strict)          */
    float tau2;        /* verification threshold, Eq. 3: re-mask iff p(current) < tau2 (strict) */
    int32_t mask_id;   /* the [MASK] token id, in [0, V)                                         */
    int32_t n_seq;     /* sequences in the batch                                                 */
    int32_t seq_len;   /* S: length of each row of `tokens`                                      */
    int32_t blk_start; /* first position of the current block Y_cur                             */
    int32_t blk_len;   /* L_b, 1..1024; blk_start + blk_len <= seq_len                           */
    int32_t max_steps; /* step budget per block for loop drivers (wino_decode); unused elsewhere */
    int32_t options;   /* bit set of WINO_OPT_* below; 0 = plain Eq. 4 on every sequence        */
    int32_t step_index;   /* k, the index of the state this step produces (Y^(k)); see last_change */
    int32_t *last_change; /* optional device int32 [n_seq, seq_len]: every position whose token the
                             step changes gets step_index.  Started at 0 and carried through a whole
                             decode with step_index = 1, 2, ..., it ends as each position's WINO
                             finalization step t_l = min{t : y_l^(j) = y_l^final for all j >= t}
                             (Sec. 5.1; 0 for the prompt).  NULL: not recorded. */
    int32_t draft_m;   /* 0: drafting by Eq. 2 (tau1 plus the at-least-one rule).  M > 0: naive
                          parallel sampling, the fixed-step-size decoding WINO is compared with
                          (Sec. 3, Sec. 6.3.3): the min(M, #MASK) masked positions with the largest
                          max_v p are drafted (smallest position first on equal confidence) and
                          tau1 is not used; M = 1 is high-confidence greedy decoding (Eq. 1).
                          Verification is unchanged; combine with WINO_OPT_NO_SHADOW for the
                          irreversible baseline decoders.  Must be >= 0. */
    const int32_t *active_seq; /* optional device int32 [n_active] (wino_step only): the sequences this
                          step scores and updates, each in [0, n_seq), no repeats.  H keeps its full
                          layout for all n_seq sequences; the step gathers the listed sequences' rows
                          (with WINO_OPT_COMPACT only the row each position reads) into the workspace
                          and scores those alone; every other sequence's tokens, counts and flags are
                          left as they are.  A batched decode lists the sequences whose block still
                          has a MASK: the others' loops have ended (as WINO_OPT_FREEZE_FINISHED), so
                          their rows need not be scored.  NULL: every sequence. */
    int32_t n_active;  /* entries of active_seq, 1..n_seq, when active_seq is not NULL */
} wino_params;

/*
 * WINO_OPT_FREEZE_FINISHED: a sequence whose current block holds no MASK
 * before the step is finished -- the per-sequence loop of Sec. 4.2.3 stops
 * there -- and is left unchanged (counts {0, 0, 0}, flags 0).  Batched decode
 * loops set it so that sequences that finish early are not re-verified while
 * they wait for the rest of the batch.
 */
#define WINO_OPT_FREEZE_FINISHED 1

/*
 * WINO_OPT_NO_SHADOW: WINO+ inference (Sec. 5.3, Sec. 6.1.2).  The model was
 * trained to follow WINO's order, so decoding drops the shadow block and
 * verification: each sequence contributes only its blk_len block rows (row
 * index s*blk_len + l, N = n_seq*blk_len), a masked position is drafted iff
 * its confidence exceeds tau1 (the single threshold; the at-least-one rule
 * still applies), and nothing is re-masked (tau2 is ignored).
 */
#define WINO_OPT_NO_SHADOW 2

/*
 * WINO_OPT_COMPACT (wino_step only): Eq. 4 reads, per position, only the
 * block row of a masked position (Eq. 2) and only the shadow row of a
 * decoded one (Eq. 3).  With this option the step first gathers that one row
 * per position into the workspace and scores n_seq*blk_len rows instead of
 * 2*n_seq*blk_len; the token state, counts and flags are those of the full
 * step.  H keeps the full [s][kind][l] layout; the workspace must hold
 * wino_workspace_size_step() bytes.
 */
#define WINO_OPT_COMPACT 4

/*
 * WINO_OPT_W_PANELS (wino_step, wino_step_static_scratch, wino_decode): the
 * W argument is the panel copy of the LM head written by
 * wino_lm_head_panels(), not the row-major [V, d] matrix (d then a multiple
 * of 64 and (d/64)*V at most 2^30, else WINO_ERR_SHAPE).  The results are
 * bit-identical to those with row-major W.
 */
#define WINO_OPT_W_PANELS 8

/*
 * Bytes of scratch wino_score_rows needs for N rows of dimension d over a
 * vocabulary of V entries, with or without the entropy output: status words,
 * per-sequence tickets, per-row partial softmax records (R = min(ceil(V/128),
 * 256) of 16 bytes per row, plus R floats per row only used for the entropy)
 * and the per-row results.  Without an entropy output the call needs R * 4 * N
 * bytes (rounded to 256) less.  `ws` must be 256-byte aligned and zero-filled
 * before its first use (for example with cudaMemsetAsync); the library keeps
 * its status words consistent from then on, so a workspace is reused as it is.
 * Returns WINO_ERR_SHAPE for sizes the kernels do not support, see
 * wino_score_rows.
 */
WINO_API int wino_workspace_size(int64_t N, int64_t d, int64_t V, size_t *bytes);

/*
 * Workspace bytes wino_step needs for these parameters (row layout,
 * WINO_OPT_COMPACT and an active-sequence list taken into account): the
 * scratch of wino_score_rows without entropy for the rows it scores, plus
 * 2*d bytes per scored row for the gathered rows of WINO_OPT_COMPACT or an
 * active-sequence list (and 4 bytes per row for their targets with a list).
 * With active_seq set, the size depends on n_active only: a workspace sized
 * for n_active = n_seq serves every list.  Zero-filled before first use, as
 * for wino_workspace_size.
 */
WINO_API int wino_workspace_size_step(const wino_params *p, int64_t d, int64_t V, size_t *bytes);

/*
 * The LM head re-laid out in d/64 panels of 64 columns (a weight layout of
 * this library; the paper has no counterpart):
 *     Wp[k][v][c] = W[v][64k + c],  k < d/64, v < V, c < 64,
 * bf16, V*d*2 bytes (the size of W).  A step with WINO_OPT_W_PANELS reads W
 * through this copy: every copy of the score kernel (bn/2 vocabulary rows x
 * one 64-wide K slice, 15-16 KB) is then one contiguous block of HBM instead
 * of bn/2 pieces of 128 bytes, 2*d bytes apart, and the W stream runs closer
 * to the HBM peak (about 2 % faster steps at one 256-row block, 1 % at
 * N = 2048).  Make the copy once per LM head and keep it while W does not
 * change; the library does not track W.
 *   W   [V, d] bf16 (uint16_t bits), device, 16-byte aligned; not modified
 *   Wp  device, 16-byte aligned, V*d*2 bytes, not overlapping W; written
 *       asynchronously on `stream`
 * d must be a multiple of 64 and (d/64)*V at most 2^30.  Returns WINO_ERR_ARG
 * for null, misaligned or overlapping buffers, WINO_ERR_SHAPE for other sizes,
 * WINO_ERR_CUDA if the launch fails.
 */
WINO_API int wino_lm_head_panels(const uint16_t *W, int64_t d, int64_t V, uint16_t *Wp, void *stream);

/*
 * Fused LM-head GEMM + full-vocabulary softmax statistics (the p_theta(.|Y~)
 * of Eq. 2 and Eq. 3), without writing the [N, V] logits anywhere.
 *   H       [N, d] bf16, row-major, 16-byte aligned      (hidden states)
 *   W       [V, d] bf16, row-major, 16-byte aligned      (LM-head weights)
 *   target  [N] int32 or NULL: token whose probability is wanted per row;
 *           a value outside [0, V) means "none"
 *   argmax  [N] int32 out: argmax_v l_v, the smallest v among exact ties
 *   pmax    [N] float out: max_v p_v = 1 / sum_v exp(l_v - max_u l_u)
 *   ptarget [N] float out: p_target, 0 where the row has no target
 *   entropy [N] float out or NULL: H(p) = -sum_v p_v ln p_v, the per-row
 *           quantity WINO+'s deferral and sharpening terms use (Sec. 5.3,
 *           Eq. 6-7); NULL skips it (the decode path never computes it)
 * Shapes: 1 <= N <= 2^24, 8 <= d <= 65536 with d % 8 == 0, 2 <= V <= 2^27.
 * Logits are accumulated in fp32 on the tensor cores; the softmax runs in
 * fp32.  ws_bytes must be at least wino_workspace_size(N, d, V) with an
 * entropy output and R * 4 * N bytes less without one (see there).
 */
WINO_API int wino_score_rows(const uint16_t *H, const uint16_t *W, int64_t N, int64_t d, int64_t V,
                    const int32_t *target, int32_t *argmax, float *pmax, float *ptarget, float *entropy,
                    void *ws, size_t ws_bytes, void *stream);

/*
 * Eq. 4 on every sequence's current block, in place on tokens[n_seq, seq_len]
 * (int32), from per-row statistics in [s][kind][l] order (argmax/pmax of the
 * kind-0 rows drive drafting; ptarget of the kind-1 rows, i.e. the
 * probability of the position's CURRENT token, drives verification).  With
 * WINO_OPT_NO_SHADOW the rows are [s][l] block rows only and ptarget may be
 * NULL.
 *   counts [n_seq, 3] int32 out: {drafted (MASK -> token), re-masked,
 *                                MASKs left in the block after the step}
 *   flags  [n_seq, blk_len] int8 out or NULL: per position 0 unchanged,
 *          1 drafted (pmax > tau1), 2 drafted by the at-least-one rule,
 *          3 re-masked, 4 selected for drafting but its argmax is MASK itself
 *          (the position stays MASK and is not counted as drafted),
 *          5 drafted by the fixed-M rule (draft_m > 0)
 * Ties in the at-least-one rule go to the smallest position.  Requires
 * 0 <= tau1, tau2 <= 1, 1 <= blk_len <= 1024, n_seq >= 1, draft_m >= 0 and
 * active_seq == NULL (the rows are the caller's).
 */
WINO_API int wino_draft_verify(int32_t *tokens, const int32_t *argmax, const float *pmax, const float *ptarget,
                      const wino_params *p, int32_t *counts, int8_t *flags, void *stream);

/*
 * One whole WINO step: targets of the shadow rows are gathered from `tokens`
 * (the current token of each decoded position, none for masked positions and
 * for block rows), every row is scored as in wino_score_rows, and Eq. 4 is
 * applied as in wino_draft_verify.
 *   H [2*n_seq*blk_len, d] bf16 rows in [s][kind][l] order (with
 *     WINO_OPT_NO_SHADOW: [n_seq*blk_len, d], block rows only); W [V, d] bf16,
 *     or with WINO_OPT_W_PANELS its panel copy (wino_lm_head_panels).
 * If a device wait expired, tokens are left unchanged and every counts entry
 * is set to WINO_ERR_DEVICE_TIMEOUT.
 */
WINO_API int wino_step(const uint16_t *H, const uint16_t *W, int64_t d, int64_t V, int32_t *tokens, const wino_params *p,
              int32_t *counts, int8_t *flags, void *ws, size_t ws_bytes, void *stream);

/*
 * wino_step without a caller-supplied workspace, for callers that cannot
 * allocate device memory: an inference-server plugin that is handed only its
 * input and output buffers, a process whose memory pool owns all device
 * memory, or a decode loop that must not call cudaMalloc / cudaFree while it
 * runs (both synchronise the device).  (The paper has no counterpart: this is
 * an interface choice of this library.)
 *
 * Same arguments, kernels and results as wino_step, with the workspace taken
 * from one fixed array of WINO_STATIC_SCRATCH_BYTES in device memory that the
 * library reserves on every GPU that loads it, until the process exits.  The
 * call allocates nothing.  A problem is accepted iff
 * wino_workspace_size_step(p, d, V) <= WINO_STATIC_SCRATCH_BYTES, and
 * rejected otherwise with WINO_ERR_WORKSPACE before anything is launched.
 * Each scored row needs R * 16 + 14 bytes, R = min(ceil(V/128), 256), so for
 * V > 32640 (R = 256): up to 4080 scored rows (N = 2 * n_seq * blk_len,
 * any d); with WINO_OPT_COMPACT or an active-sequence list the gathered rows
 * add 2*d bytes per scored row: at d = 4096, up to 1363 scored rows
 * (n_seq * blk_len with WINO_OPT_COMPACT).
 * Every call looks up the array's device address with the device current
 * (cudaGetSymbolAddress); the first call on a device also clears the status
 * words at the start of the array on `stream` (cudaMemsetAsync), so make that
 * first call before any stream capture.  Every call on a device shares the
 * one array: calls that may overlap on the GPU (different streams, or host
 * threads without ordering) race and must be serialised by the caller.  The
 * array keeps the last call's contents; the kernels clear what they rely on
 * (tickets, status words) as each call goes, and the per-row statistics it
 * holds are not returned.
 */
#define WINO_STATIC_SCRATCH_BYTES (16u << 20)
WINO_API int wino_step_static_scratch(const uint16_t *H, const uint16_t *W, int64_t d, int64_t V, int32_t *tokens,
                                      const wino_params *p, int32_t *counts, int8_t *flags, void *stream);

/*
 * Semi-autoregressive WINO decode (Sec. 3 and Sec. 4.2.3) run by the library:
 * blocks first_block .. n_blocks-1 are decoded left to right, block b starting
 * at position p->blk_start + b * p->blk_len; each block is stepped with
 * wino_step until none of its positions is MASK in any sequence.  The
 * hidden states of every step come from the caller (the transformer forward
 * with the shadow-block attention mask is outside this library):
 *   hidden(user, k, blk_start) returns the device bf16 rows of global step k
 *   for the block at blk_start, laid out as wino_step's H, and must stay
 *   valid until the next call of `hidden` or the return of wino_decode;
 *   NULL stops the decode with WINO_ERR_ARG.
 * Step k (counted from first_step) produces state Y^(k+1): it runs with
 * p->step_index = k + 1 (see last_change).  After every step the [n_seq, 3]
 * counts are copied to counts_host (host memory, pinned for speed) and the
 * stream is synchronised to decide whether the block is done: this call
 * blocks the calling thread.  p->options apply to every step; batched
 * decodes want WINO_OPT_FREEZE_FINISHED.  A block that is still not done
 * after p->max_steps (>= 1) steps returns WINO_ERR_MAX_STEPS; a device
 * failure returns its status (tokens then hold the last good state).
 *   active_buf   device int32 [n_seq] or NULL: when given, every step lists in
 *                it the sequences whose current block still has a MASK and
 *                scores only those (see wino_params.active_seq; p->active_seq
 *                itself must be NULL); ws must then be sized for n_active =
 *                n_seq.  With WINO_OPT_FREEZE_FINISHED (which it implies for the
 *                sequences it leaves out) the same states as without it.
 *   block_stats  host [n_blocks] or NULL: per block {steps, drafted, re-masked,
 *                drafted by the at-least-one rule, sequences stepped summed
 *                over the steps} (entries before first_block untouched; the
 *                at-least-one count needs flags and flags_host)
 *   flags_host   host [n_seq, blk_len] or NULL: with flags, each step's flags
 *                are copied here and the at-least-one drafts counted
 *   next_step    host or NULL: the global index after the last step run;
 *                with the block that follows, the point to resume from
 * W (row-major, or the panel copy with WINO_OPT_W_PANELS), counts, flags
 * (optional), ws and ws_bytes are as for wino_step.
 */
typedef const uint16_t *(*wino_hidden_fn)(void *user, int32_t step, int32_t blk_start);
typedef struct {
    int32_t steps, drafted, remasked, fallback;
    int32_t seq_steps; /* sequences stepped, summed over the block's steps */
} wino_block_stats;
WINO_API int wino_decode(const uint16_t *W, int64_t d, int64_t V, int32_t *tokens, const wino_params *p,
                         int32_t n_blocks, int32_t first_block, int32_t first_step, wino_hidden_fn hidden,
                         void *user, int32_t *counts, int32_t *counts_host, int8_t *flags, int8_t *flags_host,
                         int32_t *active_buf, void *ws, size_t ws_bytes, void *stream,
                         wino_block_stats *block_stats, int32_t *next_step);

/*
 * Waits for `stream`, then reads the outcome of the last call that used `ws`
 * (published by its last kernel): WINO_OK, WINO_ERR_DEVICE_TIMEOUT (a bounded
 * wait expired), WINO_ERR_ARG (an active-sequence list entry out of range) or
 * WINO_ERR_UNSUPPORTED (the TMEM allocation check failed).
 */
WINO_API int wino_read_device_status(const void *ws, void *stream, int *device_status);

/*
 * Launch timing of the fused score kernel (for benchmarks).  Between
 * wino_profile_begin(max_launches) and wino_profile_end, each of the first
 * max_launches score launches (from wino_score_rows or wino_step) is
 * bracketed by two CUDA events recorded on its stream; wino_profile_end
 * waits for the last of them and returns the summed kernel time in
 * milliseconds and the number of launches timed.  The events are created by
 * begin and destroyed by end.  Only one profile may be open per process.
 */
WINO_API int wino_profile_begin(int max_launches);
WINO_API int wino_profile_end(double *score_ms_total, int *score_launches);

/*
 * Timeline of the score kernel (diagnostics; the paper has no counterpart).
 * Between wino_timeline_begin and wino_timeline_end, score launch i (from
 * wino_score_rows or wino_step, counted from begin) writes, per CTA c, eight
 * 64-bit words at buf[((i % n_launches) * ctas_per_launch + c) * 8]:
 * %globaltimer stamps in ns of [0] kernel entry, [1] set-up done (barriers,
 * tensor memory), [2] first tensor copy issued, [3] wait for the previous
 * kernel done, [4] last MMA completed (leader CTA of a pair) or last tile
 * read (the other CTA), [5] all roles done, [6] exit; and [7] = SM id << 32
 * | tiles of the CTA pair (leader CTA).  Stamps [0], [1], [2], [5] and [6]
 * come from one thread and are ordered; [3] and [4] come from other warps,
 * whose %globaltimer readings were seen to disagree with it by up to a few
 * microseconds, so compare those only with each other or across CTAs.
 * A launch with more CTAs than ctas_per_launch writes nothing.  buf is a
 * device buffer of n_launches * ctas_per_launch * 8 uint64 owned by the
 * caller; end returns how many launches were counted.  One timeline per
 * process at a time.
 */
WINO_API int wino_timeline_begin(uint64_t *buf, int64_t n_launches, int64_t ctas_per_launch);
WINO_API int wino_timeline_end(int64_t *launches);

/*
 * How a score launch of N rows over V entries is split on the current device
 * (diagnostics; the paper has no counterpart): plan (host int32[8]) receives
 * the tile width bn, the vocabulary tiles n_vt = ceil(V / bn), the 256-row
 * blocks n_mb, the row-block groups, the CTA pairs per group G (= records per
 * row), the grid size in CTAs, 1 if the kernel works in passes (each staged
 * slice feeds both accumulators: two row blocks of a group share a tile's W
 * slice, or a row block left without a partner shares its H slice between two
 * tiles) else 0, and the shared-memory ring stages.  Pair c of the launch
 * serves row blocks c % groups (+ groups, ...) and, within each, tiles
 * c / groups (+ G, ...).
 */
WINO_API int wino_score_plan(int64_t N, int64_t d, int64_t V, int32_t *plan);

/*
 * The same work split for a device with sm_count SMs of which max_pairs CTA
 * pairs of the score kernel can be resident (152 and 76 on a GB300), without
 * touching any device (capacity planning, host-side tests).  plan (host
 * int32[10]) receives the eight fields of wino_score_plan, then the bytes of
 * one ring stage and the partial records the workspace holds per row.
 */
WINO_API int wino_score_plan_host(int64_t N, int64_t d, int64_t V, int32_t sm_count, int32_t max_pairs,
                                  int32_t *plan);

/*
 * Self-test of the failure path (device-side timeout handling; the paper has
 * no counterpart).  Enqueues one small kernel that waits, with the library's
 * bounded wait shortened to limit_ns (1 us .. 1 s), on a barrier nothing
 * arrives on; it gives up, writes WINO_ERR_DEVICE_TIMEOUT to *status (device
 * int32) and exits normally, leaving the context usable.
 */
WINO_API int wino_selftest_wait_timeout(int32_t *status, int64_t limit_ns, void *stream);

/* Static description of a status code. */
WINO_API const char *wino_status_string(int status);

/* Library version, (major << 16) | minor. */
WINO_API int wino_version(void);

#ifdef __cplusplus
}
#endif

#endif /* WINO_H */
