// wino_abi.cu -- the extern "C" entry points of libwino.so (see include/wino.h).
//
// Host side only: argument and shape checks, workspace layout, TMA tensor-map
// encoding (cached), and kernel launches on the caller's stream.  No entry
// point allocates device memory or synchronises, except
// wino_read_device_status, which reads the status words back.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>

#include <cudaTypedefs.h>  // PFN_cuTensorMapEncodeTiled

#include "internal.h"
#include "trace.h"

namespace wino {
namespace {

constexpr int64_t kMaxN = int64_t(1) << 24;
constexpr int64_t kMaxD = 65536;
constexpr int64_t kMaxV = int64_t(1) << 27;
constexpr int64_t kMaxPanelRows = int64_t(1) << 30;  // (d/64) * V of a panel copy: its row coordinates stay in int32
constexpr size_t kAlign = 256;

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Workspace layout: [status words | tickets[ceil(N/2)] | partial records [N][R] | argmax[N] | pmax[N] |
// ptarget[N] || entropy partials [N][R]], R = records_per_row(V) bounds the records per row.  `total` ends
// before the entropy partials, which only wino_score_rows with an entropy output needs (`total_entropy`).
struct WsLayout {
    size_t status, tickets, part, argmax, pmax, ptarget, total, part_u, total_entropy;
};

WsLayout ws_layout(int64_t N, int64_t V)
{
    const int64_t R = records_per_row(V);
    WsLayout L{};
    L.status = 0;
    L.tickets = kAlign;
    L.part = L.tickets + round_up((size_t)((N + 1) / 2) * 4, kAlign);
    L.argmax = L.part + round_up((size_t)N * (size_t)R * sizeof(float4), kAlign);
    L.pmax = L.argmax + round_up((size_t)N * 4, kAlign);
    L.ptarget = L.pmax + round_up((size_t)N * 4, kAlign);
    L.total = L.ptarget + round_up((size_t)N * 4, kAlign);
    L.part_u = L.total;
    L.total_entropy = L.part_u + round_up((size_t)N * (size_t)R * sizeof(float), kAlign);
    return L;
}
static_assert(sizeof(StatusWords) <= kAlign, "status words must fit the first 256 bytes");

bool shape_ok(int64_t N, int64_t d, int64_t V)
{
    return N >= 1 && N <= kMaxN && d >= 8 && d <= kMaxD && d % 8 == 0 && V >= 2 && V <= kMaxV;
}

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// ---------------------------------------------------------------- device facts

struct DeviceInfo {
    int sm_count = 0;
    bool supported = false;
};

int device_info(DeviceInfo *out)
{
    static std::mutex mu;
    static DeviceInfo cache[64];
    static bool have[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64)
        return WINO_ERR_CUDA;
    std::lock_guard<std::mutex> g(mu);
    if (!have[dev]) {
        int major = 0, minor = 0, sms = 0;
        if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            return WINO_ERR_CUDA;
        cache[dev].sm_count = sms;
        cache[dev].supported = (major == 10 && minor == 3);
        have[dev] = true;
    }
    *out = cache[dev];
    return out->supported ? WINO_OK : WINO_ERR_UNSUPPORTED;
}

// ---------------------------------------------------------------- tensor maps

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// A bf16 row-major [rows, cols] matrix read in boxes of box_rows x 64 with
// 128-byte swizzling; out-of-range rows/columns read as zero.
struct MapKey {
    const void *ptr;
    int64_t rows, cols;
    int box_rows;
    int dev;
    bool operator==(const MapKey &o) const
    {
        return ptr == o.ptr && rows == o.rows && cols == o.cols && box_rows == o.box_rows && dev == o.dev;
    }
};

int tensor_map(const void *ptr, int64_t rows, int64_t cols, int box_rows, CUtensorMap *out)
{
    static std::mutex mu;
    constexpr int kSlots = 32;
    static MapKey keys[kSlots];
    static CUtensorMap maps[kSlots];
    static int next = 0;
    int dev = 0;
    cudaGetDevice(&dev);
    const MapKey key{ptr, rows, cols, box_rows, dev};
    std::lock_guard<std::mutex> g(mu);
    for (int i = 0; i < kSlots; ++i)
        if (keys[i] == key) {
            *out = maps[i];
            return WINO_OK;
        }
    auto fn = encode_fn();
    if (!fn)
        return WINO_ERR_CUDA;
    CUtensorMap m;
    std::memset(&m, 0, sizeof m);
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(&m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return WINO_ERR_CUDA;
    keys[next] = key;
    maps[next] = m;
    next = (next + 1) % kSlots;
    *out = m;
    return WINO_OK;
}

// ---------------------------------------------------------------- score-kernel timeline (diagnostics)

// While enabled, score launch i writes its per-CTA stamps into slot i % n_launches of the caller's buffer.
struct Timeline {
    std::mutex mu;
    uint64_t *buf = nullptr;
    int64_t n_launches = 0, ctas_per_launch = 0, next = 0;
} g_timeline;

uint64_t *timeline_slot(unsigned grid)
{
    std::lock_guard<std::mutex> g(g_timeline.mu);
    if (!g_timeline.buf || (int64_t)grid > g_timeline.ctas_per_launch)
        return nullptr;
    const int64_t i = g_timeline.next++ % g_timeline.n_launches;
    return g_timeline.buf + i * g_timeline.ctas_per_launch * kTimelineWords;
}

// ---------------------------------------------------------------- launch timing

// Optional timing of the score kernel: while enabled, every score launch is
// bracketed by a pair of CUDA events recorded on the launch stream.
struct Profiler {
    std::mutex mu;
    bool on = false;
    int cap = 0, n = 0;
    cudaEvent_t *ev = nullptr;
} g_prof;

void prof_record(int which, cudaStream_t stream)
{
    if (!g_prof.on)
        return;
    std::lock_guard<std::mutex> g(g_prof.mu);
    if (!g_prof.on || g_prof.n >= g_prof.cap)
        return;
    cudaEventRecord(g_prof.ev[2 * g_prof.n + which], stream);
    if (which == 1)
        ++g_prof.n;
}

// ---------------------------------------------------------------- shared pieces

int check_params(const wino_params *p)
{
    if (!p)
        return WINO_ERR_ARG;
    if (!(p->tau1 >= 0.f && p->tau1 <= 1.f) || !(p->tau2 >= 0.f && p->tau2 <= 1.f) || p->draft_m < 0)
        return WINO_ERR_ARG;
    if (!aligned(p->last_change, 4) || !aligned(p->active_seq, 4))
        return WINO_ERR_ARG;
    if (p->active_seq && (p->n_active < 1 || p->n_active > p->n_seq))
        return WINO_ERR_SHAPE;
    if (p->n_seq < 1 || p->blk_len < 1 || p->blk_len > kMaxBlkLen || p->blk_start < 0 || p->seq_len < 1 ||
        (int64_t)p->blk_start + p->blk_len > p->seq_len || p->mask_id < 0)
        return WINO_ERR_SHAPE;
    if ((int64_t)p->n_seq * 2 * p->blk_len > kMaxN || (int64_t)p->n_seq * p->seq_len > (int64_t(1) << 31))
        return WINO_ERR_SHAPE;
    return WINO_OK;
}

// Score N rows into (argmax, pmax, ptarget), and with `step` also apply Eq. 4:
// the score kernel followed by the finish kernel.
// W is row-major [V, d], or with w_panels the panel copy [d/64][V][64] of wino_lm_head_panels.
int score_and_finish(const uint16_t *H, const uint16_t *W, bool w_panels, int64_t N, int64_t d, int64_t V,
                     const TargetSource &ts, int32_t *argmax, float *pmax, float *ptarget, float *entropy, void *ws,
                     size_t ws_bytes, const wino_params *step, int32_t *tokens, int32_t *counts, int8_t *flags,
                     cudaStream_t stream)
{
    DeviceInfo info;
    int rc = device_info(&info);
    if (rc != WINO_OK)
        return rc;
    const WsLayout L = ws_layout(N, V);
    if (ws_bytes < (entropy ? L.total_entropy : L.total))
        return WINO_ERR_WORKSPACE;
    const int max_pairs = score_max_pairs();
    if (max_pairs < 1)
        return WINO_ERR_CUDA;
    const int32_t n_mb = (int32_t)((N + kPairM - 1) / kPairM);
    const ScoreSchedule sch =
        score_schedule(n_mb, V, std::min(max_pairs, info.sm_count / 2), (int32_t)records_per_row(V));
    CUtensorMap tmH, tmW;
    if ((rc = tensor_map(H, N, d, kBM, &tmH)) != WINO_OK)
        return rc;
    // one 16-byte-aligned map row per (K slice, vocabulary row) of the panel copy
    if ((rc = w_panels ? tensor_map(W, d / kBK * V, kBK, sch.bn / 2, &tmW) : tensor_map(W, V, d, sch.bn / 2, &tmW)) !=
        WINO_OK)
        return rc;
    uint8_t *w8 = static_cast<uint8_t *>(ws);
    ScoreArgs a{};
    a.N = (int32_t)N;
    a.d = (int32_t)d;
    a.V = (int32_t)V;
    a.n_mb = n_mb;
    a.n_vt = sch.n_vt;
    a.n_kb = (int32_t)((d + kBK - 1) / kBK);
    a.bn = sch.bn;
    a.two = sch.two;
    a.stages = sch.stages;
    a.stage_bytes = sch.stage_bytes;
    a.n_groups = sch.n_groups;
    a.G = sch.G;
    a.ts = ts;
    a.part = reinterpret_cast<float4 *>(w8 + L.part);
    a.part_u = entropy ? reinterpret_cast<float *>(w8 + L.part_u) : nullptr;
    a.status = reinterpret_cast<StatusWords *>(w8 + L.status);
    a.tickets = reinterpret_cast<int32_t *>(w8 + L.tickets);
    a.n_tickets = step ? step->n_seq : 0;
    a.timeline = timeline_slot((unsigned)(2 * a.n_groups * a.G));
    a.w_panels = w_panels ? 1 : 0;
    prof_record(0, stream);
    if (launch_score(tmH, tmW, a, entropy != nullptr, stream) != cudaSuccess)
        return WINO_ERR_CUDA;
    prof_record(1, stream);
    FinishArgs f{};
    f.part = a.part;
    f.part_u = a.part_u;
    f.entropy = entropy;
    f.G = a.G;
    f.N = a.N;
    f.V = a.V;
    f.ts = ts;
    f.status = a.status;
    f.argmax = argmax;
    f.pmax = pmax;
    f.ptarget = ptarget;
    if (step) {
        f.tokens = tokens;
        f.p = *step;
        f.counts = counts;
        f.flags = flags;
        f.tickets = a.tickets;
    }
    if (launch_finish(f, stream) != cudaSuccess)
        return WINO_ERR_CUDA;
    return WINO_OK;
}

// Rows wino_step scores for these parameters, and the workspace it needs.
int64_t step_rows(const wino_params &p)
{
    const bool one_row = (p.options & (WINO_OPT_NO_SHADOW | WINO_OPT_COMPACT)) != 0;
    return (int64_t)(p.active_seq ? p.n_active : p.n_seq) * (one_row ? 1 : 2) * p.blk_len;
}

size_t step_ws_bytes(const wino_params &p, int64_t d, int64_t V)
{
    const int64_t rows = step_rows(p);
    size_t total = ws_layout(rows, V).total;
    if ((p.options & WINO_OPT_COMPACT) || p.active_seq)
        total += round_up((size_t)rows * (size_t)d * 2, kAlign);  // the gathered rows
    if (p.active_seq)
        total += round_up((size_t)rows * 4, kAlign);  // and their targets
    return total;
}

}  // namespace
}  // namespace wino

using namespace wino;

extern "C" {

int wino_version(void) { return (0 << 16) | 1; }

const char *wino_status_string(int status)
{
    switch (status) {
    case WINO_OK: return "ok";
    case WINO_ERR_ARG: return "invalid argument (null or misaligned pointer, threshold outside [0, 1])";
    case WINO_ERR_SHAPE: return "unsupported shape";
    case WINO_ERR_WORKSPACE: return "workspace too small";
    case WINO_ERR_CUDA: return "CUDA call or kernel launch failed";
    case WINO_ERR_MAX_STEPS: return "decode loop exceeded its step budget";
    case WINO_ERR_DEVICE_TIMEOUT: return "a bounded device-side wait expired; outputs are invalid";
    case WINO_ERR_UNSUPPORTED: return "device is not compute capability 10.3";
    default: return "unknown status";
    }
}

int wino_workspace_size(int64_t N, int64_t d, int64_t V, size_t *bytes)
{
    if (!bytes)
        return WINO_ERR_ARG;
    if (!shape_ok(N, d, V))
        return WINO_ERR_SHAPE;
    *bytes = ws_layout(N, V).total_entropy;
    return WINO_OK;
}

int wino_workspace_size_step(const wino_params *p, int64_t d, int64_t V, size_t *bytes)
{
    if (!p || !bytes)
        return WINO_ERR_ARG;
    if (!shape_ok(step_rows(*p), d, V))
        return WINO_ERR_SHAPE;
    *bytes = step_ws_bytes(*p, d, V);
    return WINO_OK;
}

int wino_score_rows(const uint16_t *H, const uint16_t *W, int64_t N, int64_t d, int64_t V, const int32_t *target,
                    int32_t *argmax, float *pmax, float *ptarget, float *entropy, void *ws, size_t ws_bytes,
                    void *stream)
{
    const Range range("wino_score_rows");
    if (!H || !W || !argmax || !pmax || !ptarget || !ws)
        return WINO_ERR_ARG;
    if (!aligned(H, 16) || !aligned(W, 16) || !aligned(ws, kAlign))
        return WINO_ERR_ARG;
    if (!aligned(target, 4) || !aligned(argmax, 4) || !aligned(pmax, 4) || !aligned(ptarget, 4) ||
        !aligned(entropy, 4))
        return WINO_ERR_ARG;  // 32-bit elements: a misaligned pointer would fault on the device
    if (!shape_ok(N, d, V))
        return WINO_ERR_SHAPE;
    TargetSource ts{};
    ts.target = target;
    return score_and_finish(H, W, false, N, d, V, ts, argmax, pmax, ptarget, entropy, ws, ws_bytes, nullptr, nullptr,
                            nullptr, nullptr, static_cast<cudaStream_t>(stream));
}

int wino_draft_verify(int32_t *tokens, const int32_t *argmax, const float *pmax, const float *ptarget,
                      const wino_params *p, int32_t *counts, int8_t *flags, void *stream)
{
    const Range range("wino_draft_verify");
    if (!tokens || !argmax || !pmax || !counts || !p || (!ptarget && !(p->options & WINO_OPT_NO_SHADOW)) ||
        p->active_seq)
        return WINO_ERR_ARG;
    if (!aligned(tokens, 4) || !aligned(argmax, 4) || !aligned(pmax, 4) || !aligned(ptarget, 4) ||
        !aligned(counts, 4))
        return WINO_ERR_ARG;
    int rc = check_params(p);
    if (rc != WINO_OK)
        return rc;
    DeviceInfo info;
    if ((rc = device_info(&info)) != WINO_OK)
        return rc;
    if (launch_draft_verify(tokens, argmax, pmax, ptarget, *p, counts, flags, static_cast<cudaStream_t>(stream)) !=
        cudaSuccess)
        return WINO_ERR_CUDA;
    return WINO_OK;
}

int wino_step(const uint16_t *H, const uint16_t *W, int64_t d, int64_t V, int32_t *tokens, const wino_params *p,
              int32_t *counts, int8_t *flags, void *ws, size_t ws_bytes, void *stream)
{
    const Range range("wino_step");
    if (!H || !W || !tokens || !counts || !ws)
        return WINO_ERR_ARG;
    if (!aligned(H, 16) || !aligned(W, 16) || !aligned(ws, kAlign) || !aligned(tokens, 4) || !aligned(counts, 4))
        return WINO_ERR_ARG;
    int rc = check_params(p);
    if (rc != WINO_OK)
        return rc;
    const bool shadow = !(p->options & WINO_OPT_NO_SHADOW);
    const bool compact = (p->options & WINO_OPT_COMPACT) != 0;
    if (compact && !shadow)
        return WINO_ERR_ARG;  // without a shadow block there is nothing to compact
    const int64_t N = step_rows(*p);  // rows scored
    if (!shape_ok(N, d, V) || p->mask_id >= V)
        return WINO_ERR_SHAPE;
    const bool w_panels = (p->options & WINO_OPT_W_PANELS) != 0;
    if (w_panels && (d % kBK != 0 || d / kBK * V > kMaxPanelRows))
        return WINO_ERR_SHAPE;
    const WsLayout L = ws_layout(N, V);
    if (ws_bytes < step_ws_bytes(*p, d, V))
        return WINO_ERR_WORKSPACE;
    uint8_t *w8 = static_cast<uint8_t *>(ws);
    int32_t *am = reinterpret_cast<int32_t *>(w8 + L.argmax);
    float *pm = reinterpret_cast<float *>(w8 + L.pmax);
    float *pt = reinterpret_cast<float *>(w8 + L.ptarget);
    TargetSource ts{};
    ts.tokens = shadow ? tokens : nullptr;  // only shadow rows have targets
    ts.seq_len = p->seq_len;
    ts.blk_start = p->blk_start;
    ts.blk_len = p->blk_len;
    ts.mask_id = p->mask_id;
    ts.compact = compact ? 1 : 0;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const uint16_t *Hs = H;
    if (p->active_seq) {  // gather the listed sequences' rows (and their targets) behind the workspace proper
        DeviceInfo info;
        if ((rc = device_info(&info)) != WINO_OK)
            return rc;
        uint16_t *Hc = reinterpret_cast<uint16_t *>(w8 + L.total);
        int32_t *tgt = reinterpret_cast<int32_t *>(w8 + L.total + round_up((size_t)N * (size_t)d * 2, kAlign));
        if (launch_gather_active(H, Hc, tgt, tokens, *p, N, d, s) != cudaSuccess)
            return WINO_ERR_CUDA;
        TargetSource tsa{};
        tsa.target = tgt;
        return score_and_finish(Hc, W, w_panels, N, d, V, tsa, am, pm, pt, nullptr, ws, ws_bytes, p, tokens, counts,
                                flags, s);
    }
    if (compact) {  // gather the one row per position Eq. 4 reads, behind the workspace proper
        DeviceInfo info;
        if ((rc = device_info(&info)) != WINO_OK)
            return rc;
        uint16_t *Hc = reinterpret_cast<uint16_t *>(w8 + L.total);
        if (launch_gather_compact(H, Hc, tokens, *p, d, s) != cudaSuccess)
            return WINO_ERR_CUDA;
        Hs = Hc;
    }
    return score_and_finish(Hs, W, w_panels, N, d, V, ts, am, pm, pt, nullptr, ws, ws_bytes, p, tokens, counts, flags,
                            s);
}

int wino_lm_head_panels(const uint16_t *W, int64_t d, int64_t V, uint16_t *Wp, void *stream)
{
    const Range range("wino_lm_head_panels");
    if (!W || !Wp || !aligned(W, 16) || !aligned(Wp, 16))
        return WINO_ERR_ARG;
    if (d < kBK || d > kMaxD || d % kBK != 0 || V < 2 || V > kMaxV || d / kBK * V > kMaxPanelRows)
        return WINO_ERR_SHAPE;
    const uintptr_t bytes = (uintptr_t)V * (uintptr_t)d * 2u;
    const uintptr_t w0 = reinterpret_cast<uintptr_t>(W), p0 = reinterpret_cast<uintptr_t>(Wp);
    if (w0 < p0 + bytes && p0 < w0 + bytes)
        return WINO_ERR_ARG;  // the copy cannot be made in place
    DeviceInfo info;
    int rc = device_info(&info);
    if (rc != WINO_OK)
        return rc;
    if (launch_panels(W, Wp, d, V, info.sm_count, static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return WINO_ERR_CUDA;
    return WINO_OK;
}

int wino_profile_begin(int max_launches)
{
    if (max_launches < 1 || max_launches > (1 << 20))
        return WINO_ERR_ARG;
    std::lock_guard<std::mutex> g(g_prof.mu);
    if (g_prof.on)
        return WINO_ERR_ARG;
    g_prof.ev = new cudaEvent_t[2 * (size_t)max_launches];
    for (int i = 0; i < 2 * max_launches; ++i)
        if (cudaEventCreate(&g_prof.ev[i]) != cudaSuccess) {
            for (int j = 0; j < i; ++j)
                cudaEventDestroy(g_prof.ev[j]);
            delete[] g_prof.ev;
            g_prof.ev = nullptr;
            return WINO_ERR_CUDA;
        }
    g_prof.cap = max_launches;
    g_prof.n = 0;
    g_prof.on = true;
    return WINO_OK;
}

int wino_profile_end(double *score_ms_total, int *score_launches)
{
    if (!score_ms_total || !score_launches)
        return WINO_ERR_ARG;
    std::lock_guard<std::mutex> g(g_prof.mu);
    if (!g_prof.on)
        return WINO_ERR_ARG;
    int rc = WINO_OK;
    double total = 0.0;
    for (int i = 0; i < g_prof.n; ++i) {
        float ms = 0.f;
        if (cudaEventSynchronize(g_prof.ev[2 * i + 1]) != cudaSuccess ||
            cudaEventElapsedTime(&ms, g_prof.ev[2 * i], g_prof.ev[2 * i + 1]) != cudaSuccess)
            rc = WINO_ERR_CUDA;
        total += ms;
    }
    for (int i = 0; i < 2 * g_prof.cap; ++i)
        cudaEventDestroy(g_prof.ev[i]);
    delete[] g_prof.ev;
    g_prof.ev = nullptr;
    *score_ms_total = total;
    *score_launches = g_prof.n;
    g_prof.on = false;
    g_prof.cap = g_prof.n = 0;
    return rc;
}

int wino_read_device_status(const void *ws, void *stream, int *device_status)
{
    if (!ws || !device_status)
        return WINO_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess)
        return WINO_ERR_CUDA;
    StatusWords w{};
    if (cudaMemcpy(&w, ws, sizeof w, cudaMemcpyDeviceToHost) != cudaSuccess)
        return WINO_ERR_CUDA;
    *device_status = w.last;
    return WINO_OK;
}

int wino_score_plan_host(int64_t N, int64_t d, int64_t V, int32_t sm_count, int32_t max_pairs, int32_t *plan)
{
    if (!plan || sm_count < 2 || max_pairs < 1)
        return WINO_ERR_ARG;
    if (!shape_ok(N, d, V))
        return WINO_ERR_SHAPE;
    const int32_t n_mb = (int32_t)((N + kPairM - 1) / kPairM);
    const ScoreSchedule sch =
        score_schedule(n_mb, V, std::min(max_pairs, sm_count / 2), (int32_t)records_per_row(V));
    plan[0] = sch.bn;
    plan[1] = sch.n_vt;
    plan[2] = n_mb;
    plan[3] = sch.n_groups;
    plan[4] = sch.G;
    plan[5] = 2 * sch.n_groups * sch.G;
    plan[6] = sch.two;
    plan[7] = sch.stages;
    plan[8] = (int32_t)sch.stage_bytes;
    plan[9] = (int32_t)records_per_row(V);
    return WINO_OK;
}

int wino_score_plan(int64_t N, int64_t d, int64_t V, int32_t *plan)
{
    if (!plan)
        return WINO_ERR_ARG;
    if (!shape_ok(N, d, V))
        return WINO_ERR_SHAPE;
    DeviceInfo info;
    int rc = device_info(&info);
    if (rc != WINO_OK)
        return rc;
    const int max_pairs = score_max_pairs();
    if (max_pairs < 1)
        return WINO_ERR_CUDA;
    const int32_t n_mb = (int32_t)((N + kPairM - 1) / kPairM);
    const ScoreSchedule sch =
        score_schedule(n_mb, V, std::min(max_pairs, info.sm_count / 2), (int32_t)records_per_row(V));
    plan[0] = sch.bn;
    plan[1] = sch.n_vt;
    plan[2] = n_mb;
    plan[3] = sch.n_groups;
    plan[4] = sch.G;
    plan[5] = 2 * sch.n_groups * sch.G;
    plan[6] = sch.two;
    plan[7] = sch.stages;
    return WINO_OK;
}

int wino_timeline_begin(uint64_t *buf, int64_t n_launches, int64_t ctas_per_launch)
{
    if (!buf || !aligned(buf, 8) || n_launches < 1 || ctas_per_launch < 2 || ctas_per_launch > (1 << 16) ||
        n_launches > (int64_t(1) << 20))
        return WINO_ERR_ARG;
    std::lock_guard<std::mutex> g(g_timeline.mu);
    if (g_timeline.buf)
        return WINO_ERR_ARG;
    g_timeline.buf = buf;
    g_timeline.n_launches = n_launches;
    g_timeline.ctas_per_launch = ctas_per_launch;
    g_timeline.next = 0;
    return WINO_OK;
}

int wino_timeline_end(int64_t *launches)
{
    if (!launches)
        return WINO_ERR_ARG;
    std::lock_guard<std::mutex> g(g_timeline.mu);
    if (!g_timeline.buf)
        return WINO_ERR_ARG;
    *launches = g_timeline.next;
    g_timeline.buf = nullptr;
    g_timeline.n_launches = g_timeline.ctas_per_launch = g_timeline.next = 0;
    return WINO_OK;
}

}  // extern "C"
