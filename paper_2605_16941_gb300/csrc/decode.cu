// decode.cu -- the semi-autoregressive decode loop (Sec. 3 and Sec. 4.2.3) run by the library.
//
// Blocks are decoded left to right; inside a block wino_step is repeated until
// no position of the block is MASK in any sequence.  The hidden states of each
// step come from a caller callback (the transformer forward is outside this
// library); after each step the [n_seq, 3] counts are copied to the caller's
// host buffer and the stream is synchronised, because whether the block is done
// is only known once the step has run.  With an active-sequence buffer the loop
// also keeps the list of sequences whose block still has a MASK and steps only
// those (the others' loops have ended).  The loop is host code only: every
// launch goes through wino_step.
#include <vector>

#include <cuda_runtime.h>

#include "trace.h"
#include "wino.h"

extern "C" int wino_decode(const uint16_t *W, int64_t d, int64_t V, int32_t *tokens, const wino_params *p,
                           int32_t n_blocks, int32_t first_block, int32_t first_step, wino_hidden_fn hidden,
                           void *user, int32_t *counts, int32_t *counts_host, int8_t *flags, int8_t *flags_host,
                           int32_t *active_buf, void *ws, size_t ws_bytes, void *stream,
                           wino_block_stats *block_stats, int32_t *next_step)
{
    const wino::Range range("wino_decode");
    if (!W || !tokens || !p || !hidden || !counts || !counts_host || !ws || (flags_host && !flags) || p->active_seq)
        return WINO_ERR_ARG;
    if (n_blocks < 1 || first_block < 0 || first_block > n_blocks || first_step < 0 || p->max_steps < 1)
        return WINO_ERR_ARG;
    if (p->n_seq < 1 || p->blk_len < 1 || p->blk_start < 0 ||
        (int64_t)p->blk_start + (int64_t)n_blocks * p->blk_len > (int64_t)p->seq_len)
        return WINO_ERR_SHAPE;  // every block must lie inside the sequence
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int32_t n_seq = p->n_seq;
    const size_t count_bytes = (size_t)n_seq * 3 * sizeof(int32_t);
    const size_t flag_bytes = (size_t)n_seq * p->blk_len;
    std::vector<int32_t> active(n_seq), still;  // sequences stepped (host copy of active_buf)
    still.reserve(n_seq);
    wino_params q = *p;
    int32_t k = first_step;
    int rc = WINO_OK;
    for (int32_t b = first_block; b < n_blocks && rc == WINO_OK; ++b) {
        q.blk_start = p->blk_start + b * p->blk_len;
        wino_block_stats bs{0, 0, 0, 0, 0};
        int32_t n_active = n_seq;  // a new block: every sequence takes part
        for (int32_t i = 0; i < n_seq; ++i)
            active[i] = i;
        for (;;) {
            if (bs.steps >= p->max_steps) {
                rc = WINO_ERR_MAX_STEPS;
                break;
            }
            const uint16_t *H = hidden(user, k, q.blk_start);
            if (!H) {
                rc = WINO_ERR_ARG;
                break;
            }
            q.step_index = k + 1;  // this step produces state Y^(k+1)
            if (active_buf) {
                if (cudaMemcpyAsync(active_buf, active.data(), (size_t)n_active * sizeof(int32_t),
                                    cudaMemcpyHostToDevice, s) != cudaSuccess) {
                    rc = WINO_ERR_CUDA;
                    break;
                }
                q.active_seq = active_buf;
                q.n_active = n_active;
            }
            rc = wino_step(H, W, d, V, tokens, &q, counts, flags, ws, ws_bytes, stream);
            if (rc != WINO_OK)
                break;
            if (cudaMemcpyAsync(counts_host, counts, count_bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
                (flags_host && cudaMemcpyAsync(flags_host, flags, flag_bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess) ||
                cudaStreamSynchronize(s) != cudaSuccess) {
                rc = WINO_ERR_CUDA;
                break;
            }
            // Only the sequences stepped have fresh counts and flags.
            still.clear();
            for (int32_t ai = 0; ai < n_active; ++ai) {
                const int32_t i = active[ai];
                const int32_t *c = counts_host + 3 * i;
                if (c[0] < 0 || c[1] < 0 || c[2] < 0) {  // a device failure: the state was left alone
                    rc = c[0] < 0 ? c[0] : (c[1] < 0 ? c[1] : c[2]);
                    break;
                }
                bs.drafted += c[0];
                bs.remasked += c[1];
                if (flags_host)
                    for (int32_t l = 0; l < p->blk_len; ++l)
                        bs.fallback += (flags_host[(size_t)i * p->blk_len + l] == 2);  // at-least-one drafts
                if (c[2] != 0)
                    still.push_back(i);
            }
            if (rc != WINO_OK)
                break;
            ++k;
            ++bs.steps;
            bs.seq_steps += n_active;
            if (still.empty())
                break;  // no sequence has a MASK left in this block
            if (active_buf) {
                n_active = (int32_t)still.size();
                for (int32_t ai = 0; ai < n_active; ++ai)
                    active[ai] = still[ai];
            }
        }
        if (block_stats)
            block_stats[b] = bs;
    }
    if (next_step)
        *next_step = k;
    return rc;
}
