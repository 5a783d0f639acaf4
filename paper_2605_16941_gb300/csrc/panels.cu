// panels.cu -- the LM head's panel layout (wino_lm_head_panels): Wp[k][v][c] = W[v][64k + c].
//
// The score kernel reads W in copies of bn/2 vocabulary rows x one 64-wide K slice.  In row-major W such a
// copy is bn/2 pieces of 128 B, 2*d bytes apart; in the panel copy it is one contiguous block.  The copy is made
// once per LM head, so this kernel is a plain grid-stride loop over 16-byte pieces: consecutive threads write
// consecutive pieces of Wp (coalesced) and read 128-byte runs of W rows.
#include <cstdint>

#include "internal.h"

namespace wino {
namespace {

__global__ void panels_kernel(const uint4 *__restrict__ W, uint4 *__restrict__ Wp, int32_t V, int32_t n_kb)
{
    // piece i of Wp: 16 bytes c8 (of 8) of row v in panel k, i = (k * V + v) * 8 + c8
    const int64_t total = (int64_t)n_kb * V * 8;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int32_t c8 = (int32_t)(i & 7);
        const int32_t kv = (int32_t)(i >> 3);  // k * V + v, below 2^30
        const int32_t k = kv / V, v = kv - k * V;
        Wp[i] = W[((int64_t)v * n_kb + k) * 8 + c8];
    }
}

}  // namespace

cudaError_t launch_panels(const uint16_t *W, uint16_t *Wp, int64_t d, int64_t V, int sm_count, cudaStream_t stream)
{
    constexpr int kThreads = 256;
    const int64_t pieces = V * d / 8;
    int64_t blocks = (pieces + kThreads - 1) / kThreads;
    const int64_t cap = (int64_t)sm_count * 8;  // a few waves of the grid-stride loop
    if (blocks > cap)
        blocks = cap;
    panels_kernel<<<(unsigned)blocks, kThreads, 0, stream>>>(reinterpret_cast<const uint4 *>(W),
                                                              reinterpret_cast<uint4 *>(Wp), (int32_t)V,
                                                              (int32_t)(d / 64));
    return cudaGetLastError();
}

}  // namespace wino
