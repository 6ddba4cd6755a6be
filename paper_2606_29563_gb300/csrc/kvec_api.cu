// C ABI of the K-VEC eviction-selection library: validation, workspace, launch
// sequence.  Declarations and the meaning of every argument are in kvec.h.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <string>
#include <vector>

#include "kvec.h"
#include "kvec_internal.cuh"

using namespace kvec;

namespace {

thread_local std::string g_last_error;

kvec_status fail(kvec_status s, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return s;
}

kvec_status cuda_fail(cudaError_t e, const char* what) {
    return fail(KVEC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Row stride of per-position workspace arrays: 128-byte aligned rows with room for
// a float4 access that starts at the last position of a row.
size_t row_stride(int max_seqlen) { return round_up((size_t)max_seqlen + 4, 32); }

constexpr int kKernelKinds = 5;

// Fault injected for tests of the error path (kvec_set_test_fault); 0 = none.
std::atomic<int> g_test_fault{0};

// Maps a device error word to a status (and the message of kvec_last_error).
kvec_status device_error_status(int err) {
    if (err == 2)
        return fail(KVEC_ERR_INVALID_ARG,
                    "a call would have taken a coverage state past 255 layers (that state was left unchanged)");
    return fail(KVEC_ERR_DEVICE_TIMEOUT, "a bounded device wait gave up (code %d)", err);
}

struct TimedLaunch {
    int kind;
    cudaEvent_t start, stop;
};

}  // namespace

int kvec::test_fault() { return g_test_fault.load(std::memory_order_relaxed); }

constexpr int kSlots = 8;   // per-layer score arrays in flight between the score and select stages
constexpr int kScoreBufs = 2;   // segment-partial buffers in flight between the score and row-statistics stages
constexpr size_t kGraphCache = 16;  // captured multi-layer calls kept per handle

struct kvec_handle {
    kvec_params p;
    int device = 0;
    int num_sms = 1;
    int g = 1, R = 0, words = 0;
    size_t state_stride = 0, n_off = 16, union_off = 0;
    void* ws = nullptr;
    size_t ws_bytes = 0;
    int* claims = nullptr;   // [max_layers] the score launches' chunk counters (zero between launches)
    Scratch sc{};
    Scratch score_buf[kScoreBufs]{};   // segment partials, one per layer in flight
    Slot slots[kSlots]{};
    float2* rowstat_slot[kSlots]{};    // row statistics of the layer in slot k (read by its window grid)
    int last_slot = 0;
    int last_batch = 0;
    bool profiling = false;
    std::vector<TimedLaunch> timed;
    std::vector<cudaEvent_t> event_pool;
    // Streams of the layer pipeline: score | window | heads (two, alternating by
    // layer, so consecutive layers' head passes overlap) | coverage select | gather.
    cudaStream_t s_score = nullptr, s_win = nullptr, s_heads = nullptr, s_heads2 = nullptr, s_chain = nullptr,
                 s_gather = nullptr, s_cap = nullptr;
    std::vector<cudaEvent_t> ev_score, ev_rs, ev_win, ev_heads, ev_sel, ev_gather;
    cudaEvent_t ev_fork = nullptr, ev_join[5] = {nullptr, nullptr, nullptr, nullptr, nullptr};
    // Scheduling priorities: the heads and coverage-select kernels (the serial
    // chain of the pipeline) take SMs before the score, window and gather kernels.
    int prio_hi = 0, prio_lo = 0;
    // CUDA graph of the last repeated multi-layer call.
    // Captured graphs of repeated multi-layer calls, most recent last (at most
    // kGraphCache), and the keys of calls seen once (a second sighting captures).
    struct CachedGraph {
        std::vector<uint64_t> key;
        cudaGraphExec_t exec;
    };
    std::vector<CachedGraph> graphs;
    std::vector<std::vector<uint64_t>> seen_keys;
    // While a call is captured: each programmatic launch's graph node and the
    // node of the kernel before it on the same stream (null if none), whose edge
    // alone may stay programmatic (restore_full_edges).
    bool capturing = false;
    std::vector<std::pair<cudaGraphNode_t, cudaGraphNode_t>> prog_nodes;
};

namespace {

cudaEvent_t take_event(kvec_handle* h) {
    if (!h->event_pool.empty()) {
        cudaEvent_t e = h->event_pool.back();
        h->event_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}

void recycle_timed(kvec_handle* h) {
    for (auto& t : h->timed) {
        h->event_pool.push_back(t.start);
        h->event_pool.push_back(t.stop);
    }
    h->timed.clear();
}

template <class F>
void timed_launch(kvec_handle* h, int kind, cudaStream_t st, F&& launch) {
    if (!h->profiling) {
        launch();
        return;
    }
    TimedLaunch t{kind, take_event(h), take_event(h)};
    cudaEventRecord(t.start, st);
    launch();
    cudaEventRecord(t.stop, st);
    h->timed.push_back(t);
}

kvec_status validate_params(const kvec_params* p) {
    if (!p) return fail(KVEC_ERR_INVALID_ARG, "params is NULL");
    if (p->num_kv_heads < 1 || p->num_q_heads < p->num_kv_heads || p->num_q_heads % p->num_kv_heads)
        return fail(KVEC_ERR_INVALID_ARG, "num_q_heads (%d) must be a positive multiple of num_kv_heads (%d)",
                    p->num_q_heads, p->num_kv_heads);
    if (p->num_kv_heads > 32)
        return fail(KVEC_ERR_UNSUPPORTED, "num_kv_heads > 32 is not supported (a token's KV heads share one warp)");
    if (p->head_dim != kHeadDim) return fail(KVEC_ERR_UNSUPPORTED, "head_dim must be %d", kHeadDim);
    if (p->window < 1) return fail(KVEC_ERR_INVALID_ARG, "window must be >= 1");
    if (p->obs_window < 1 || p->obs_window > p->window || p->ext_window < 1 || p->ext_window > p->window)
        return fail(KVEC_ERR_INVALID_ARG, "need 1 <= obs_window, ext_window <= window");
    if (p->obs_window > kMaxObsWindow)
        return fail(KVEC_ERR_UNSUPPORTED, "obs_window > %d is not supported", kMaxObsWindow);
    const int g = p->num_q_heads / p->num_kv_heads;
    if ((g * p->window) % 8 != 0 || g * p->window > 256)
        return fail(KVEC_ERR_UNSUPPORTED, "rows per KV head (group %d x window %d) must be a multiple of 8 and <= 256",
                    g, p->window);
    if (p->pool_kernel < 1 || p->pool_kernel > kMaxPool || p->pool_kernel % 2 == 0)
        return fail(KVEC_ERR_INVALID_ARG, "pool_kernel must be odd and in [1, %d]", kMaxPool);
    if (p->pool_mode != 0 && p->pool_mode != 1) return fail(KVEC_ERR_INVALID_ARG, "pool_mode must be 0 or 1");
    if (p->head_criterion != 0 && p->head_criterion != 1)
        return fail(KVEC_ERR_INVALID_ARG, "head_criterion must be 0 or 1");
    if (p->all_positions != 0 && p->all_positions != 1)
        return fail(KVEC_ERR_INVALID_ARG, "all_positions must be 0 or 1");
    if (p->num_ext_heads < 0 || p->num_ext_heads > p->num_kv_heads)
        return fail(KVEC_ERR_INVALID_ARG, "num_ext_heads must be in [0, num_kv_heads]");
    if (!(p->beta >= 0.f && p->beta <= 1.f)) return fail(KVEC_ERR_INVALID_ARG, "beta must be in [0, 1]");
    if (!isfinite(p->lambda)) return fail(KVEC_ERR_INVALID_ARG, "lambda must be finite");
    if (!isfinite(p->softmax_scale)) return fail(KVEC_ERR_INVALID_ARG, "softmax_scale must be finite");
    if (p->max_batch < 1 || p->max_seqlen < 1 || p->max_seqlen > 131072)
        return fail(KVEC_ERR_INVALID_ARG, "need max_batch >= 1 and 1 <= max_seqlen <= 131072");
    if (p->max_layers < 1 || p->max_layers > 255)
        return fail(KVEC_ERR_INVALID_ARG, "max_layers must be in [1, 255]");
    if (p->head_budget != 0 && p->head_budget != 1) return fail(KVEC_ERR_INVALID_ARG, "head_budget must be 0 or 1");
    if (p->head_budget && !(p->ada_floor >= 0.f && p->ada_floor <= 1.f))
        return fail(KVEC_ERR_INVALID_ARG, "ada_floor must be in [0, 1]");
    return KVEC_OK;
}

// Preserved tokens K, fill F = B - wk - K and the fill a head ranks itself.
void budget_split(const kvec_params& p, int budget, int* Kp, int* F, int* f0) {
    const int wk = p.all_positions ? 0 : p.window;
    int k = (int)floor((double)p.beta * (double)budget);
    if (k > budget - wk) k = budget - wk;
    *Kp = k;
    *F = budget - wk - k;
    *f0 = p.head_budget ? (int)floor((double)p.ada_floor * (double)*F) : *F;
}

kvec_status set_device(kvec_handle* h, int* prev) {
    cudaError_t e = cudaGetDevice(prev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (*prev != h->device) {
        e = cudaSetDevice(h->device);
        if (e != cudaSuccess) return cuda_fail(e, "cudaSetDevice");
    }
    return KVEC_OK;
}

struct DeviceGuard {
    int prev, dev;
    ~DeviceGuard() {
        if (prev != dev) cudaSetDevice(prev);
    }
};

kvec_status validate_call(kvec_handle* h, int batch, const int32_t* cu_host, const int32_t* cu_dev, int budget,
                          int* total_tiles, int* total_win_tiles) {
    if (!h) return fail(KVEC_ERR_INVALID_ARG, "handle is NULL");
    if (batch < 1 || batch > h->p.max_batch)
        return fail(KVEC_ERR_INVALID_ARG, "batch %d outside [1, max_batch=%d]", batch, h->p.max_batch);
    if (!cu_host || !cu_dev) return fail(KVEC_ERR_INVALID_ARG, "cu_seqlens pointers must not be NULL");
    if (cu_host[0] != 0) return fail(KVEC_ERR_INVALID_ARG, "cu_seqlens[0] must be 0");
    const int wk = h->p.all_positions ? 0 : h->p.window;   // the tail kept unconditionally
    if (budget < 1) return fail(KVEC_ERR_INVALID_ARG, "budget %d < 1", budget);
    if (budget < wk) return fail(KVEC_ERR_INVALID_ARG, "budget %d < window %d", budget, wk);
    int tiles = 0, chunks = 0;
    for (int b = 0; b < batch; ++b) {
        const int L = cu_host[b + 1] - cu_host[b];
        if (L < h->p.window || L > h->p.max_seqlen)
            return fail(KVEC_ERR_INVALID_ARG, "sequence %d has length %d outside [window=%d, max_seqlen=%d]", b, L,
                        h->p.window, h->p.max_seqlen);
        tiles += (L + kTileT - 1) / kTileT;
        chunks += (L - wk + kTileT - 1) / kTileT;   // candidate tiles of the window kernel
    }
    *total_tiles = tiles;
    *total_win_tiles = chunks;
    return KVEC_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

constexpr int kDecodeMaxCap = 1 << 20;   // cached rows per (sequence, KV head) a decode call may pass

Geometry make_geometry(const kvec_handle* h, int batch, int budget, int tiles, int chunks, int total_tokens) {
    const kvec_params& p = h->p;
    Geometry G{};
    G.Hq = p.num_q_heads;
    G.Hkv = p.num_kv_heads;
    G.g = h->g;
    G.w = p.window;
    G.O = p.obs_window;
    G.Oe = p.ext_window;
    G.pool = p.pool_kernel;
    G.pool_avg = p.pool_mode;
    G.head_entropy = p.head_criterion;
    G.delta = p.num_ext_heads;
    G.R = h->R;
    G.lambda = p.lambda;
    const double scale = p.softmax_scale > 0.f ? (double)p.softmax_scale : 1.0 / sqrt((double)p.head_dim);
    G.sl2 = (float)(scale * 1.4426950408889634);
    G.ML = (int)row_stride(p.max_seqlen);
    G.words = h->words;
    G.batch = batch;
    G.budget = budget;
    G.wk = p.all_positions ? 0 : p.window;
    budget_split(p, budget, &G.Kp, &G.k2, &G.f0);
    G.ada = p.head_budget;
    G.extras = p.num_kv_heads * (G.k2 - G.f0);
    G.cap = budget + (p.num_kv_heads - 1) * (G.k2 - G.f0);
    G.jpool = G.ada ? std::min(G.extras, 32 * G.words) : 0;
    G.jstride = p.num_kv_heads * G.ML + 32;
    G.total_tiles = tiles;
    G.win_tiles = chunks;
    G.HG = p.num_kv_heads < kWinHeadsPerCta ? p.num_kv_heads : kWinHeadsPerCta;
    G.NG = (p.num_kv_heads + G.HG - 1) / G.HG;
    G.total_tokens = total_tokens;
    G.state_stride = h->state_stride;
    G.state_n_off = h->n_off;
    G.state_union_off = h->union_off;
    G.nlen = (int)round_up((size_t)p.max_seqlen, 16);
    return G;
}

// One layer, every kernel on one stream with one slot (used without a handle).
kvec_status run_layer_sequential(kvec_handle* h, const Geometry& G, const LayerIO& io, cudaStream_t st) {
    ScorePlan plan;
    cudaError_t se = plan_score(G, io, h->sc, h->num_sms, &plan);
    if (se != cudaSuccess) return cuda_fail(se, "score kernel tensor maps");
    se = launch_score(plan, h->claims, st, false);
    if (se != cudaSuccess) return cuda_fail(se, "score kernel launch");
    se = launch_rowstat(plan, G, io, h->sc, h->claims, st, /*programmatic=*/true, /*after_score=*/true);
    if (se != cudaSuccess) return cuda_fail(se, "row statistics launch");
    se = launch_window(plan, G, io, h->sc, h->slots[0], st, false);
    if (se != cudaSuccess) return cuda_fail(se, "window kernel launch");
    se = launch_heads(G, io, h->sc, h->slots[0], st, h->prio_hi);
    if (se != cudaSuccess) return cuda_fail(se, "heads kernel launch");
    se = launch_select(G, io, h->sc, h->slots[0], nullptr, st, h->prio_hi, 0, 1, /*programmatic=*/false);
    if (se != cudaSuccess) return cuda_fail(se, "select kernel launch");
    launch_gather(G, io, h->slots[0], st);
    se = launch_finalize(G, io, h->sc, h->slots[0], st, h->prio_hi, 1);
    if (se != cudaSuccess) return cuda_fail(se, "finalize kernel launch");
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "kernel launch");
    return KVEC_OK;
}

// The node a capturing stream added last (its only current dependency), or null
// when the stream is not capturing.
cudaGraphNode_t captured_tail(cudaStream_t st) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    const cudaGraphNode_t* deps = nullptr;
    const cudaGraphEdgeData* ed = nullptr;
    size_t nd = 0;
    if (cudaStreamGetCaptureInfo(st, &cs, nullptr, nullptr, &deps, &ed, &nd) != cudaSuccess) return nullptr;
    return (cs == cudaStreamCaptureStatusActive && nd == 1) ? deps[0] : nullptr;
}

// Stream capture gives a programmatic launch's every incoming edge the
// programmatic type, the edges from other streams' event waits included, and
// such an edge lets the kernel start (and read) before that producer has
// finished.  Launched eagerly, only the edge from the same stream's previous
// kernel is relaxed.  This puts the captured graph back in that form: every
// other programmatic edge into a recorded node becomes a full dependency.
cudaError_t restore_full_edges(cudaGraph_t graph, const std::vector<std::pair<cudaGraphNode_t, cudaGraphNode_t>>& nodes) {
    for (const auto& nd : nodes) {
        cudaGraphNode_t node = nd.first;
        size_t n = 0;
        cudaError_t e = cudaGraphNodeGetDependencies(node, nullptr, nullptr, &n);
        if (e != cudaSuccess && e != cudaErrorLossyQuery) return e;
        std::vector<cudaGraphNode_t> deps(n);
        std::vector<cudaGraphEdgeData> ed(n);
        if (n > 0) {
            e = cudaGraphNodeGetDependencies(node, deps.data(), ed.data(), &n);
            if (e != cudaSuccess) return e;
        }
        for (size_t i = 0; i < n; ++i) {
            if (deps[i] == nd.second) continue;
            if (ed[i].type == cudaGraphDependencyTypeDefault && ed[i].from_port == 0 && ed[i].to_port == 0) continue;
            e = cudaGraphRemoveDependencies(graph, &deps[i], &node, &ed[i], 1);
            if (e != cudaSuccess) return e;
            cudaGraphEdgeData full = {};
            e = cudaGraphAddDependencies(graph, &deps[i], &node, &full, 1);
            if (e != cudaSuccess) return e;
        }
    }
    return cudaSuccess;
}

#define KV_CHECK(call)                                        \
    do {                                                      \
        cudaError_t e_ = (call);                              \
        if (e_ != cudaSuccess) return cuda_fail(e_, #call);   \
    } while (0)

// Layers 0..n-1 as a five-stream pipeline.  Only the coverage-adjusted select
// is serial across layers (it carries n_t); the score, window and heads work of
// later layers runs ahead of it, bounded by the double-buffered score scratch
// and by the kSlots ring of per-layer score arrays.  The row statistics live
// with the slot (for the window grid); a layer's score grid reuses the segment
// partials of layer l - kScoreBufs after that layer's window grid, or, when the
// score and window grids fit on the SMs together, as soon as its row
// statistics are done with them (else an early score grid only takes SMs that
// the window and heads kernels of the layers ahead need: measured slower).
// With the caller's log-sum-exp there is no score grid, and the same wait
// keeps at most two layers' window grids in flight.
kvec_status launch_pipeline(kvec_handle* h, const Geometry& G, const LayerIO* ios, int n, cudaStream_t origin) {
    KV_CHECK(cudaEventRecord(h->ev_fork, origin));
    for (cudaStream_t st : {h->s_score, h->s_win, h->s_heads, h->s_heads2, h->s_chain, h->s_gather})
        KV_CHECK(cudaStreamWaitEvent(st, h->ev_fork, 0));
    cudaGraphNode_t prev_score = nullptr, prev_window = nullptr, prev_select = nullptr;   // captured (h->capturing)
    for (int l = 0; l < n; ++l) {
        const Slot& sl = h->slots[l % kSlots];
        Scratch sc = h->score_buf[l % kScoreBufs];
        sc.rowstat = h->rowstat_slot[l % kSlots];
        const LayerIO& io = ios[l];
        ScorePlan plan;
        cudaError_t se = plan_score(G, io, sc, h->num_sms, &plan);
        if (se != cudaSuccess) return cuda_fail(se, "score kernel tensor maps");
        // Partials buffer reuse (window stream).
        if (l >= kScoreBufs) {
            const bool early = !io.lse && plan.grid + window_grid_size(plan, G, false) <= h->num_sms;
            KV_CHECK(cudaStreamWaitEvent(h->s_score, early ? h->ev_rs[l - kScoreBufs] : h->ev_win[l - kScoreBufs], 0));
        }
        // The score grid of layer l > 0 is a programmatic dependent of layer
        // l - 1's (it reads none of its results); the event wait above stays a
        // full dependency (restore_full_edges when captured).
        if (!io.lse) {
            timed_launch(h, 0, h->s_score, [&] { se = launch_score(plan, h->claims + l, h->s_score, l > 0); });
            if (se != cudaSuccess) return cuda_fail(se, "score kernel launch");
            if (h->capturing) {
                cudaGraphNode_t node = captured_tail(h->s_score);
                if (!node) return fail(KVEC_ERR_CUDA, "score kernel: no captured node");
                if (l > 0) h->prog_nodes.emplace_back(node, prev_score);
                prev_score = node;
            }
        }
        KV_CHECK(cudaEventRecord(h->ev_score[l], h->s_score));
        // Window stream: the row statistics (after the score grid and, for slot
        // reuse, after layer l - kSlots's selection and gather), then the window
        // sums as their programmatic dependent (it waits before reading them).
        KV_CHECK(cudaStreamWaitEvent(h->s_win, h->ev_score[l], 0));
        if (l >= kSlots) {
            KV_CHECK(cudaStreamWaitEvent(h->s_win, h->ev_sel[l - kSlots], 0));
            KV_CHECK(cudaStreamWaitEvent(h->s_win, h->ev_gather[l - kSlots], 0));
        }
        // The row statistics are a programmatic dependent of the previous layer's
        // window grid, which they do not wait for: they read only this layer's
        // partials (full dependency above), and the statistics buffer they
        // overwrite belongs to this layer's slot, last read by layer l - kSlots's
        // window grid (the waits above).  So consecutive window grids overlap.
        se = io.lse ? launch_rowstat_lse(G, io, sc, h->s_win, l > 0)
                    : launch_rowstat(plan, G, io, sc, h->claims + l, h->s_win, l > 0, /*after_score=*/false);
        if (se != cudaSuccess) return cuda_fail(se, "row statistics launch");
        if (h->capturing) {
            cudaGraphNode_t node = captured_tail(h->s_win);
            if (!node) return fail(KVEC_ERR_CUDA, "row statistics: no captured node");
            if (l > 0) h->prog_nodes.emplace_back(node, prev_window);
        }
        KV_CHECK(cudaEventRecord(h->ev_rs[l], h->s_win));
        timed_launch(h, 1, h->s_win, [&] { se = launch_window(plan, G, io, sc, sl, h->s_win, true); });
        if (se != cudaSuccess) return cuda_fail(se, "window kernel launch");
        if (h->capturing) {
            prev_window = captured_tail(h->s_win);
            if (!prev_window) return fail(KVEC_ERR_CUDA, "window kernel: no captured node");
        }
        KV_CHECK(cudaEventRecord(h->ev_win[l], h->s_win));
        cudaStream_t s_h = (l & 1) ? h->s_heads2 : h->s_heads;
        KV_CHECK(cudaStreamWaitEvent(s_h, h->ev_win[l], 0));
        timed_launch(h, 2, s_h, [&] { se = launch_heads(G, io, sc, sl, s_h, h->prio_hi); });
        if (se != cudaSuccess) return cuda_fail(se, "heads kernel launch");
        KV_CHECK(cudaEventRecord(h->ev_heads[l], s_h));
        KV_CHECK(cudaStreamWaitEvent(h->s_chain, h->ev_heads[l], 0));
        const Slot* prev = l > 0 ? &h->slots[(l - 1) % kSlots] : nullptr;
        // The selection is a programmatic dependent of the previous layer's: it
        // stages this layer's scores (behind the full dependency on the heads
        // kernels) while that one drains.
        timed_launch(h, 3, h->s_chain,
                     [&] { se = launch_select(G, io, sc, sl, prev, h->s_chain, h->prio_hi, l, n, /*programmatic=*/true); });
        if (se != cudaSuccess) return cuda_fail(se, "select kernel launch");
        if (h->capturing) {
            cudaGraphNode_t node = captured_tail(h->s_chain);
            if (!node) return fail(KVEC_ERR_CUDA, "select kernel: no captured node");
            h->prog_nodes.emplace_back(node, prev_select);
            prev_select = node;
        }
        if (G.ada) {
            se = launch_ada(G, io, sc, sl, h->s_chain, h->prio_hi, n);
            if (se != cudaSuccess) return cuda_fail(se, "adaptive fill launch");
            if (h->capturing) {
                cudaGraphNode_t node = captured_tail(h->s_chain);
                if (!node) return fail(KVEC_ERR_CUDA, "adaptive fill: no captured node");
                h->prog_nodes.emplace_back(node, prev_select);
                prev_select = node;
            }
        }
        KV_CHECK(cudaEventRecord(h->ev_sel[l], h->s_chain));
        KV_CHECK(cudaStreamWaitEvent(h->s_gather, h->ev_sel[l], 0));
        timed_launch(h, 4, h->s_gather, [&] { launch_gather(G, io, sl, h->s_gather); });
        KV_CHECK(cudaEventRecord(h->ev_gather[l], h->s_gather));
    }
    // The last layer's union goes into the state.
    {
        cudaError_t se = launch_finalize(G, ios[n - 1], h->score_buf[(n - 1) % kScoreBufs], h->slots[(n - 1) % kSlots], h->s_chain,
                                         h->prio_hi, n);
        if (se != cudaSuccess) return cuda_fail(se, "finalize kernel launch");
    }
    KV_CHECK(cudaGetLastError());
    KV_CHECK(cudaEventRecord(h->ev_join[0], h->s_score));
    KV_CHECK(cudaEventRecord(h->ev_join[1], h->s_win));
    KV_CHECK(cudaEventRecord(h->ev_join[2], h->s_heads));
    KV_CHECK(cudaEventRecord(h->ev_join[3], h->s_gather));
    KV_CHECK(cudaEventRecord(h->ev_join[4], h->s_heads2));
    KV_CHECK(cudaEventRecord(h->ev_fork, h->s_chain));   // reused: the end of the chain stream
    KV_CHECK(cudaStreamWaitEvent(origin, h->ev_fork, 0));
    for (cudaEvent_t e : h->ev_join) KV_CHECK(cudaStreamWaitEvent(origin, e, 0));
    h->last_slot = (n - 1) % kSlots;
    return KVEC_OK;
}

std::vector<uint64_t> graph_key(int n, int batch, int budget, const int32_t* cu_host, const int32_t* cu_dev,
                                const LayerIO* ios) {
    std::vector<uint64_t> k = {(uint64_t)n, (uint64_t)batch, (uint64_t)budget, (uint64_t)(uintptr_t)cu_dev};
    for (int b = 0; b <= batch; ++b) k.push_back((uint64_t)cu_host[b]);
    for (int l = 0; l < n; ++l) {
        const LayerIO& io = ios[l];
        for (const void* ptr : {(const void*)io.q, (const void*)io.k, (const void*)io.v, (const void*)io.state,
                                (const void*)io.out_idx, (const void*)io.out_k, (const void*)io.out_v,
                                (const void*)io.lse})
            k.push_back((uint64_t)(uintptr_t)ptr);
    }
    return k;
}

}  // namespace

namespace {

void release_handle(kvec_handle* h) {
    for (auto& g : h->graphs) cudaGraphExecDestroy(g.exec);
    h->graphs.clear();
    for (cudaStream_t st : {h->s_score, h->s_win, h->s_heads, h->s_heads2, h->s_chain, h->s_gather, h->s_cap})
        if (st) cudaStreamDestroy(st);
    for (auto* v : {&h->ev_score, &h->ev_rs, &h->ev_win, &h->ev_heads, &h->ev_sel, &h->ev_gather})
        for (cudaEvent_t ev : *v)
            if (ev) cudaEventDestroy(ev);
    if (h->ev_fork) cudaEventDestroy(h->ev_fork);
    for (cudaEvent_t ev : h->ev_join)
        if (ev) cudaEventDestroy(ev);
    recycle_timed(h);
    for (cudaEvent_t ev : h->event_pool) cudaEventDestroy(ev);
    if (h->ws) cudaFree(h->ws);
    delete h;
}

}  // namespace

extern "C" {

size_t kvec_state_bytes(int max_seqlen) {
    if (max_seqlen < 1) return 0;
    const size_t ns = round_up((size_t)max_seqlen, 16);
    const size_t words = ((size_t)max_seqlen + 31) / 32;
    return round_up(16 + ns + 4 * words, 16);
}

int kvec_output_capacity(const kvec_params* params, int budget) {
    if (validate_params(params) != KVEC_OK) return -1;
    const int wk = params->all_positions ? 0 : params->window;
    if (budget < 1 || budget < wk) return -1;
    int Kp, F, f0;
    budget_split(*params, budget, &Kp, &F, &f0);
    return budget + (params->num_kv_heads - 1) * (F - f0);
}

kvec_status kvec_create(const kvec_params* params, kvec_handle** out) {
    if (!out) return fail(KVEC_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    kvec_status s = validate_params(params);
    if (s != KVEC_OK) return s;
    kvec_handle* h = new kvec_handle();
    h->p = *params;
    cudaError_t e = cudaGetDevice(&h->device);
    if (e != cudaSuccess) {
        delete h;
        return cuda_fail(e, "cudaGetDevice");
    }
    const kvec_params& p = h->p;
    h->g = p.num_q_heads / p.num_kv_heads;
    h->R = h->g * p.window;
    h->words = (p.max_seqlen + 31) / 32;
    h->state_stride = kvec_state_bytes(p.max_seqlen);
    h->n_off = 16;
    h->union_off = 16 + round_up((size_t)p.max_seqlen, 16);

    const size_t MB = p.max_batch, ML = row_stride(p.max_seqlen), Hkv = p.num_kv_heads, R = h->R,
                 W = h->words;
    const size_t max_tiles = MB * ((ML + kTileT - 1) / kTileT);
    const size_t HGmax = Hkv < (size_t)kWinHeadsPerCta ? Hkv : (size_t)kWinHeadsPerCta;
    const size_t NGmax = (Hkv + HGmax - 1) / HGmax;
    struct Part {
        void** dst;
        size_t bytes;
    };
    std::vector<Part> parts = {

        {(void**)&h->sc.keys, MB * Hkv * ML * sizeof(uint32_t)},
        {(void**)&h->sc.nbuf, MB * round_up((size_t)p.max_seqlen, 16)},
        {(void**)&h->sc.err, sizeof(int)},
        {(void**)&h->sc.keys_sel, MB * Hkv * ML * sizeof(uint32_t)},
        {(void**)&h->sc.jkeys, p.head_budget ? MB * (Hkv * ML + 32) * sizeof(uint32_t) : 0},
        {(void**)&h->sc.jpos, p.head_budget ? MB * (Hkv * ML + 32) * sizeof(int32_t) : 0},
        {(void**)&h->sc.jbits, p.head_budget ? MB * (Hkv * ML + 32) / 32 * sizeof(uint32_t) : 0},
        {(void**)&h->claims, (size_t)p.max_layers * sizeof(int)},
    };
    for (int k = 0; k < kScoreBufs; ++k) {
        Scratch& b = h->score_buf[k];
        std::vector<Part> sp = {
            {(void**)&b.segpart, max_tiles * Hkv * R * sizeof(float2)},
        };
        parts.insert(parts.end(), sp.begin(), sp.end());
    }
    for (int k = 0; k < kSlots; ++k) {
        Slot& sl = h->slots[k];
        std::vector<Part> sp = {
            {(void**)&sl.rawO, MB * Hkv * ML * sizeof(float)},  {(void**)&sl.rawOe, MB * Hkv * ML * sizeof(float)},
            {(void**)&sl.rawI, MB * ML * sizeof(float)},        {(void**)&sl.PO, MB * Hkv * ML * sizeof(float)},
            {(void**)&sl.POe, MB * Hkv * ML * sizeof(float)},   {(void**)&sl.I, MB * ML * sizeof(float)},
            {(void**)&sl.sigma, MB * Hkv * sizeof(float)},      {(void**)&sl.htop, MB * Hkv * sizeof(int)},
            {(void**)&sl.pres, MB * Hkv * W * sizeof(uint32_t)}, {(void**)&sl.Pprime, MB * Hkv * ML * sizeof(float)},
            {(void**)&sl.sel, MB * Hkv * W * sizeof(uint32_t)},
            {(void**)&sl.wpart, max_tiles * NGmax * p.obs_window * kTileT * sizeof(float)},
            {(void**)&h->rowstat_slot[k], MB * Hkv * R * sizeof(float2)},
        };
        parts.insert(parts.end(), sp.begin(), sp.end());
    }
    size_t total = 0;
    for (auto& pt : parts) total += round_up(pt.bytes, 256);
    e = cudaMalloc(&h->ws, total);
    if (e != cudaSuccess) {
        cudaGetLastError();
        delete h;
        return fail(KVEC_ERR_OOM, "workspace of %zu bytes: %s", total, cudaGetErrorString(e));
    }
    h->ws_bytes = total;
    e = cudaMemset(h->ws, 0, total);
    size_t off = 0;
    for (auto& pt : parts) {
        *pt.dst = static_cast<char*>(h->ws) + off;
        off += round_up(pt.bytes, 256);
    }
    for (Scratch& b : h->score_buf) {
        b.keys = h->sc.keys;
        b.keys_sel = h->sc.keys_sel;
        b.jkeys = h->sc.jkeys;
        b.jpos = h->sc.jpos;
        b.jbits = h->sc.jbits;
        b.nbuf = h->sc.nbuf;
        b.err = h->sc.err;
    }
    Geometry G = make_geometry(h, 1, p.window, 1, 1, p.window);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
    if (e == cudaSuccess) e = configure_score(G);
    if (e == cudaSuccess) e = configure_window(G);
    if (e == cudaSuccess) e = configure_select();
    if (e == cudaSuccess) e = cudaDeviceGetStreamPriorityRange(&h->prio_lo, &h->prio_hi);
    for (cudaStream_t* st : {&h->s_score, &h->s_gather, &h->s_cap})
        if (e == cudaSuccess) e = cudaStreamCreateWithPriority(st, cudaStreamNonBlocking, h->prio_lo);
    // A layer's window sums go ahead of the next layer's statistics when both wait for SMs.
    if (e == cudaSuccess)
        e = cudaStreamCreateWithPriority(&h->s_win, cudaStreamNonBlocking, h->prio_hi < h->prio_lo ? h->prio_lo - 1 : h->prio_lo);
    for (cudaStream_t* st : {&h->s_heads, &h->s_heads2, &h->s_chain})
        if (e == cudaSuccess) e = cudaStreamCreateWithPriority(st, cudaStreamNonBlocking, h->prio_hi);
    h->ev_score.assign(p.max_layers, nullptr);
    h->ev_rs.assign(p.max_layers, nullptr);
    h->ev_win.assign(p.max_layers, nullptr);
    h->ev_heads.assign(p.max_layers, nullptr);
    h->ev_sel.assign(p.max_layers, nullptr);
    h->ev_gather.assign(p.max_layers, nullptr);
    for (auto* v : {&h->ev_score, &h->ev_rs, &h->ev_win, &h->ev_heads, &h->ev_sel, &h->ev_gather})
        for (auto& ev : *v)
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming);
    for (auto& ev : h->ev_join)
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        release_handle(h);
        return cuda_fail(e, "workspace set-up");
    }
    *out = h;
    return KVEC_OK;
}

kvec_status kvec_destroy(kvec_handle* h) {
    if (!h) return fail(KVEC_ERR_INVALID_ARG, "handle is NULL");
    int prev = 0;
    kvec_status s = set_device(h, &prev);
    if (s != KVEC_OK) return s;
    DeviceGuard guard{prev, h->device};
    cudaError_t e = cudaDeviceSynchronize();
    release_handle(h);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
    return KVEC_OK;
}

kvec_status kvec_reset(kvec_handle* h, void* coverage_state, int batch, kvec_stream_t stream) {
    if (!h) return fail(KVEC_ERR_INVALID_ARG, "handle is NULL");
    if (!coverage_state || batch < 1 || batch > h->p.max_batch)
        return fail(KVEC_ERR_INVALID_ARG, "coverage_state must be non-NULL and 1 <= batch <= max_batch");
    int prev = 0;
    kvec_status s = set_device(h, &prev);
    if (s != KVEC_OK) return s;
    DeviceGuard guard{prev, h->device};
    cudaError_t e = cudaMemsetAsync(coverage_state, 0, h->state_stride * (size_t)batch, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
    return KVEC_OK;
}

kvec_status kvec_select_layer(kvec_handle* h, int batch, const int32_t* cu_seqlens_host,
                              const int32_t* cu_seqlens_dev, const void* q_obs, const void* k, const void* v,
                              void* coverage_state, int budget, int32_t* out_idx, void* out_k, void* out_v,
                              kvec_stream_t stream) {
    const void* qs[1] = {q_obs};
    const void* ks[1] = {k};
    const void* vs[1] = {v};
    int32_t* ois[1] = {out_idx};
    void* oks[1] = {out_k};
    void* ovs[1] = {out_v};
    return kvec_select_layers(h, 1, batch, cu_seqlens_host, cu_seqlens_dev, qs, ks, vs, coverage_state, budget, ois,
                              oks, ovs, stream);
}

}  // extern "C"

namespace {

kvec_status select_layers_impl(kvec_handle* h, int num_layers, int batch, const int32_t* cu_seqlens_host,
                               const int32_t* cu_seqlens_dev, const void* const* q_obs, const void* const* k,
                               const void* const* v, const float* const* lse, void* coverage_state, int budget,
                               int32_t* const* out_idx, void* const* out_k, void* const* out_v,
                               kvec_stream_t stream) {
    int tiles = 0, chunks = 0;
    kvec_status s = validate_call(h, batch, cu_seqlens_host, cu_seqlens_dev, budget, &tiles, &chunks);
    if (s != KVEC_OK) return s;
    if (num_layers < 1 || num_layers > h->p.max_layers)
        return fail(KVEC_ERR_INVALID_ARG, "num_layers %d outside [1, max_layers=%d]", num_layers, h->p.max_layers);
    if (!q_obs || !k || !v || !out_idx || !out_k || !out_v || !coverage_state)
        return fail(KVEC_ERR_INVALID_ARG, "NULL pointer argument");
    if (!aligned16(coverage_state)) return fail(KVEC_ERR_INVALID_ARG, "coverage_state must be 16-byte aligned");
    for (int l = 0; l < num_layers; ++l) {
        if (!q_obs[l] || !k[l] || !v[l] || !out_idx[l] || !out_k[l] || !out_v[l])
            return fail(KVEC_ERR_INVALID_ARG, "NULL pointer for layer %d", l);
        if (!aligned16(q_obs[l]) || !aligned16(k[l]) || !aligned16(v[l]) || !aligned16(out_k[l]) ||
            !aligned16(out_v[l]) || (reinterpret_cast<uintptr_t>(out_idx[l]) & 3u))
            return fail(KVEC_ERR_INVALID_ARG, "layer %d: device pointers must be 16-byte aligned", l);
        if (lse && (!lse[l] || (reinterpret_cast<uintptr_t>(lse[l]) & 3u)))
            return fail(KVEC_ERR_INVALID_ARG, "layer %d: lse must be a non-NULL, 4-byte aligned device pointer", l);
    }
    int prev = 0;
    s = set_device(h, &prev);
    if (s != KVEC_OK) return s;
    DeviceGuard guard{prev, h->device};
    Geometry G = make_geometry(h, batch, budget, tiles, chunks, cu_seqlens_host[batch]);
    G.cu_host = cu_seqlens_host;
    cudaStream_t st = (cudaStream_t)stream;
    std::vector<LayerIO> ios(num_layers);
    for (int l = 0; l < num_layers; ++l) {
        LayerIO& io = ios[l];
        io.q = static_cast<const __nv_bfloat16*>(q_obs[l]);
        io.k = static_cast<const __nv_bfloat16*>(k[l]);
        io.v = static_cast<const __nv_bfloat16*>(v[l]);
        io.cu = cu_seqlens_dev;
        io.state = static_cast<uint8_t*>(coverage_state);
        io.out_idx = out_idx[l];
        io.out_k = static_cast<__nv_bfloat16*>(out_k[l]);
        io.out_v = static_cast<__nv_bfloat16*>(out_v[l]);
        io.lse = lse ? lse[l] : nullptr;
    }
    // Graphs are neither captured nor replayed while a test fault is injected:
    // a captured launch would keep the fault after it is switched off.
    if (!h->profiling && num_layers >= 2 && test_fault() == 0) {
        // A call repeated with the same arguments replays a captured graph of the pipeline.
        std::vector<uint64_t> key = graph_key(num_layers, batch, budget, cu_seqlens_host, cu_seqlens_dev, ios.data());
        for (size_t i = 0; i < h->graphs.size(); ++i) {
            if (h->graphs[i].key != key) continue;
            KV_CHECK(cudaGraphLaunch(h->graphs[i].exec, st));
            h->last_slot = (num_layers - 1) % kSlots;
            h->last_batch = batch;
            return KVEC_OK;
        }
        bool seen = false;
        for (const auto& k : h->seen_keys) seen = seen || k == key;
        if (seen) {
            cudaGraph_t graph = nullptr;
            KV_CHECK(cudaStreamBeginCapture(h->s_cap, cudaStreamCaptureModeThreadLocal));
            h->capturing = true;
            h->prog_nodes.clear();
            s = launch_pipeline(h, G, ios.data(), num_layers, h->s_cap);
            h->capturing = false;
            cudaError_t ce = cudaStreamEndCapture(h->s_cap, &graph);
            if (s == KVEC_OK && ce == cudaSuccess) {
                ce = restore_full_edges(graph, h->prog_nodes);
                if (ce != cudaSuccess) s = cuda_fail(ce, "graph edges of the captured pipeline");
            }
            h->prog_nodes.clear();
            if (s != KVEC_OK) {
                if (graph) cudaGraphDestroy(graph);
                return s;
            }
            if (ce != cudaSuccess) return cuda_fail(ce, "cudaStreamEndCapture");
            cudaGraphExec_t exec = nullptr;
            ce = cudaGraphInstantiateWithFlags(&exec, graph, cudaGraphInstantiateFlagUseNodePriority);
            cudaGraphDestroy(graph);
            if (ce != cudaSuccess) return cuda_fail(ce, "cudaGraphInstantiate");
            if (h->graphs.size() == kGraphCache) {
                cudaGraphExecDestroy(h->graphs.front().exec);
                h->graphs.erase(h->graphs.begin());
            }
            h->graphs.push_back({key, exec});
            KV_CHECK(cudaGraphLaunch(exec, st));
            h->last_batch = batch;
            return KVEC_OK;
        }
        if (h->seen_keys.size() == kGraphCache) h->seen_keys.erase(h->seen_keys.begin());
        h->seen_keys.push_back(key);
    }
    s = launch_pipeline(h, G, ios.data(), num_layers, st);
    if (s != KVEC_OK) return s;
    h->last_batch = batch;
    return KVEC_OK;
}

}  // namespace

extern "C" {

kvec_status kvec_select_layers(kvec_handle* h, int num_layers, int batch, const int32_t* cu_seqlens_host,
                               const int32_t* cu_seqlens_dev, const void* const* q_obs, const void* const* k,
                               const void* const* v, void* coverage_state, int budget, int32_t* const* out_idx,
                               void* const* out_k, void* const* out_v, kvec_stream_t stream) {
    return select_layers_impl(h, num_layers, batch, cu_seqlens_host, cu_seqlens_dev, q_obs, k, v, nullptr,
                              coverage_state, budget, out_idx, out_k, out_v, stream);
}

kvec_status kvec_select_layers_lse(kvec_handle* h, int num_layers, int batch, const int32_t* cu_seqlens_host,
                                   const int32_t* cu_seqlens_dev, const void* const* q_obs, const void* const* k,
                                   const void* const* v, const float* const* lse, void* coverage_state, int budget,
                                   int32_t* const* out_idx, void* const* out_k, void* const* out_v,
                                   kvec_stream_t stream) {
    if (!lse) return fail(KVEC_ERR_INVALID_ARG, "NULL pointer argument");
    return select_layers_impl(h, num_layers, batch, cu_seqlens_host, cu_seqlens_dev, q_obs, k, v, lse,
                              coverage_state, budget, out_idx, out_k, out_v, stream);
}

kvec_status kvec_select_layer_lse(kvec_handle* h, int batch, const int32_t* cu_seqlens_host,
                                  const int32_t* cu_seqlens_dev, const void* q_obs, const void* k, const void* v,
                                  const float* lse, void* coverage_state, int budget, int32_t* out_idx, void* out_k,
                                  void* out_v, kvec_stream_t stream) {
    const void* qs[1] = {q_obs};
    const void* ks[1] = {k};
    const void* vs[1] = {v};
    const float* ls[1] = {lse};
    int32_t* ois[1] = {out_idx};
    void* oks[1] = {out_k};
    void* ovs[1] = {out_v};
    return kvec_select_layers_lse(h, 1, batch, cu_seqlens_host, cu_seqlens_dev, qs, ks, vs, ls, coverage_state,
                                  budget, ois, oks, ovs, stream);
}

// ---------------------------------------------------------------------------
// kvec_select_layer_noalloc: the same layer as kvec_select_layer for callers
// that may not allocate device memory.  Its scratch lives in one file-scope
// static device array that every GPU loading this library holds until exit.
// ---------------------------------------------------------------------------
}  // extern "C"

namespace {

constexpr size_t kNoallocScratchBytes = size_t(32) << 20;   // 32 MiB
__device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

constexpr int kMaxDevices = 64;
struct NoallocDevice {
    bool ready = false;
    void* base = nullptr;   // device address of g_noalloc_scratch on that device
};
NoallocDevice g_noalloc_dev[kMaxDevices];
std::mutex g_noalloc_mutex;

// Once per device, with that device current: resolve the array's device address
// (host code cannot use the symbol's name as a pointer) and set the kernels'
// shared-memory limits.  Neither call allocates.
kvec_status noalloc_setup(int dev, void** base, const Geometry& G) {
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (dev < 0 || dev >= kMaxDevices) return fail(KVEC_ERR_UNSUPPORTED, "device index %d out of range", dev);
    NoallocDevice& d = g_noalloc_dev[dev];
    if (!d.ready) {
        void* ptr = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
        if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(scratch)");
        e = configure_score(G);
        if (e == cudaSuccess) e = configure_window(G);
        if (e == cudaSuccess) e = configure_select();
        if (e != cudaSuccess) return cuda_fail(e, "kernel attributes");
        // The error word (the array's first bytes) starts at zero; calls leave it
        // set until kvec_noalloc_sync_status reads and clears it.
        e = cudaMemset(ptr, 0, sizeof(int));
        if (e == cudaSuccess) e = cudaDeviceSynchronize();
        if (e != cudaSuccess) return cuda_fail(e, "clearing the scratch error word");
        d.base = ptr;
        d.ready = true;
    }
    *base = d.base;
    return KVEC_OK;
}

}  // namespace

extern "C" {

kvec_status kvec_select_layer_noalloc(const kvec_params* params, int batch, const int32_t* cu_seqlens_host,
                                      const int32_t* cu_seqlens_dev, const void* q_obs, const void* k,
                                      const void* v, void* coverage_state, int budget, int32_t* out_idx,
                                      void* out_k, void* out_v, kvec_stream_t stream) {
    kvec_status s = validate_params(params);
    if (s != KVEC_OK) return s;
    if (params->head_budget)
        return fail(KVEC_ERR_UNSUPPORTED, "the head-wise adaptive fill needs a handle (kvec_create)");
    // A stack handle carries the geometry; its vectors stay empty and nothing is allocated.
    kvec_handle tmp;
    tmp.p = *params;
    tmp.g = params->num_q_heads / params->num_kv_heads;
    tmp.R = tmp.g * params->window;
    tmp.words = (params->max_seqlen + 31) / 32;
    tmp.state_stride = kvec_state_bytes(params->max_seqlen);
    tmp.n_off = 16;
    tmp.union_off = 16 + round_up((size_t)params->max_seqlen, 16);
    int tiles = 0, chunks = 0;
    s = validate_call(&tmp, batch, cu_seqlens_host, cu_seqlens_dev, budget, &tiles, &chunks);
    if (s != KVEC_OK) return s;
    if (!q_obs || !k || !v || !out_idx || !out_k || !out_v || !coverage_state)
        return fail(KVEC_ERR_INVALID_ARG, "NULL pointer argument");
    if (!aligned16(q_obs) || !aligned16(k) || !aligned16(v) || !aligned16(out_k) || !aligned16(out_v) ||
        !aligned16(coverage_state) || (reinterpret_cast<uintptr_t>(out_idx) & 3u))
        return fail(KVEC_ERR_INVALID_ARG, "device pointers must be 16-byte aligned");

    // Carve the scratch for exactly this call's geometry.
    const size_t nb = batch, ML = row_stride(params->max_seqlen), Hkv = params->num_kv_heads, R = tmp.R,
                 W = tmp.words;
    const size_t nt = tiles;
    struct Part {
        void** dst;
        size_t bytes;
    };
    const size_t HGv = Hkv < (size_t)kWinHeadsPerCta ? Hkv : (size_t)kWinHeadsPerCta;
    const size_t NGv = (Hkv + HGv - 1) / HGv;
    Part parts[] = {
        {(void**)&tmp.sc.err, sizeof(int)},                   // error word, first: see noalloc_setup
        {(void**)&tmp.claims, sizeof(int)},
        {(void**)&tmp.sc.nbuf, nb * round_up((size_t)params->max_seqlen, 16)},
        {(void**)&tmp.sc.segpart, nt * Hkv * R * sizeof(float2)},
        {(void**)&tmp.slots[0].wpart, nt * NGv * (size_t)params->obs_window * kTileT * sizeof(float)},
        {(void**)&tmp.sc.rowstat, nb * Hkv * R * sizeof(float2)},
        {(void**)&tmp.sc.keys, nb * Hkv * ML * sizeof(uint32_t)},
        {(void**)&tmp.sc.keys_sel, nb * Hkv * ML * sizeof(uint32_t)},
        {(void**)&tmp.slots[0].rawO, nb * Hkv * ML * sizeof(float)},
        {(void**)&tmp.slots[0].rawOe, nb * Hkv * ML * sizeof(float)},
        {(void**)&tmp.slots[0].rawI, nb * ML * sizeof(float)},
        {(void**)&tmp.slots[0].PO, nb * Hkv * ML * sizeof(float)},
        {(void**)&tmp.slots[0].POe, nb * Hkv * ML * sizeof(float)},
        {(void**)&tmp.slots[0].I, nb * ML * sizeof(float)},
        {(void**)&tmp.slots[0].sigma, nb * Hkv * sizeof(float)},
        {(void**)&tmp.slots[0].htop, nb * Hkv * sizeof(int)},
        {(void**)&tmp.slots[0].pres, nb * Hkv * W * sizeof(uint32_t)},
        {(void**)&tmp.slots[0].Pprime, nb * Hkv * ML * sizeof(float)},
        {(void**)&tmp.slots[0].sel, nb * Hkv * W * sizeof(uint32_t)},
    };
    size_t need = 0;
    for (size_t i = 0; i < sizeof(parts) / sizeof(parts[0]); ++i) need += round_up(parts[i].bytes, 256);
    if (need > kNoallocScratchBytes)
        return fail(KVEC_ERR_INVALID_ARG,
                    "this call needs %zu bytes of scratch; kvec_select_layer_noalloc has %zu (use kvec_create / "
                    "kvec_select_layer for larger batches or sequences)",
                    need, kNoallocScratchBytes);

    int prev = 0;
    cudaError_t e = cudaGetDevice(&prev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    tmp.device = prev;
    e = cudaDeviceGetAttribute(&tmp.num_sms, cudaDevAttrMultiProcessorCount, prev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    Geometry G = make_geometry(&tmp, batch, budget, tiles, chunks, cu_seqlens_host[batch]);
    G.cu_host = cu_seqlens_host;
    void* base = nullptr;
    s = noalloc_setup(prev, &base, G);
    if (s != KVEC_OK) return s;
    size_t off = 0;
    for (auto& pt : parts) {
        *pt.dst = static_cast<char*>(base) + off;
        off += round_up(pt.bytes, 256);
    }
    cudaStream_t st = (cudaStream_t)stream;
    // The rest of the array keeps the previous call's contents: every part below
    // the error word is written before it is read within the call.
    LayerIO io{};
    io.q = static_cast<const __nv_bfloat16*>(q_obs);
    io.k = static_cast<const __nv_bfloat16*>(k);
    io.v = static_cast<const __nv_bfloat16*>(v);
    io.cu = cu_seqlens_dev;
    io.state = static_cast<uint8_t*>(coverage_state);
    io.out_idx = out_idx;
    io.out_k = static_cast<__nv_bfloat16*>(out_k);
    io.out_v = static_cast<__nv_bfloat16*>(out_v);
    return run_layer_sequential(&tmp, G, io, st);
}

kvec_status kvec_noalloc_sync_status(kvec_stream_t stream) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    void* base = nullptr;
    {
        std::lock_guard<std::mutex> lock(g_noalloc_mutex);
        if (dev >= 0 && dev < kMaxDevices && g_noalloc_dev[dev].ready) base = g_noalloc_dev[dev].base;
    }
    if (!base) return KVEC_OK;   // no call has run on this device
    e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    int err = 0;
    e = cudaMemcpy(&err, base, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "reading the scratch error word");
    if (err) {
        e = cudaMemset(base, 0, sizeof(int));
        if (e == cudaSuccess) e = cudaDeviceSynchronize();
        if (e != cudaSuccess) return cuda_fail(e, "clearing the scratch error word");
        return device_error_status(err);
    }
    return KVEC_OK;
}

kvec_status kvec_decode_attention(kvec_handle* h, int batch, const void* q, const void* k_cache,
                                  const void* v_cache, const int32_t* lens, int cap, float* out,
                                  kvec_stream_t stream) {
    if (!h) return fail(KVEC_ERR_INVALID_ARG, "handle is NULL");
    const kvec_params& p = h->p;
    if (batch < 1 || batch > p.max_batch)
        return fail(KVEC_ERR_INVALID_ARG, "batch %d outside [1, max_batch = %d]", batch, p.max_batch);
    if (cap < 1 || cap > kDecodeMaxCap)
        return fail(KVEC_ERR_INVALID_ARG, "cap %d outside [1, %d]", cap, kDecodeMaxCap);
    if (h->g > 8)
        return fail(KVEC_ERR_UNSUPPORTED, "decode attention supports up to 8 query heads per KV head (g = %d)", h->g);
    if (!q || !k_cache || !v_cache || !lens || !out) return fail(KVEC_ERR_INVALID_ARG, "a device pointer is NULL");
    if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache))
        return fail(KVEC_ERR_INVALID_ARG, "q, k_cache and v_cache must be 16-byte aligned");
    if (reinterpret_cast<uintptr_t>(lens) % 4 || reinterpret_cast<uintptr_t>(out) % 8)
        return fail(KVEC_ERR_INVALID_ARG, "lens must be 4-byte and out 8-byte aligned");
    DecodeIO io{};
    io.q = static_cast<const __nv_bfloat16*>(q);
    io.k = static_cast<const __nv_bfloat16*>(k_cache);
    io.v = static_cast<const __nv_bfloat16*>(v_cache);
    io.lens = lens;
    io.out = out;
    io.batch = batch;
    io.Hq = p.num_q_heads;
    io.Hkv = p.num_kv_heads;
    io.cap = cap;
    io.scale = p.softmax_scale > 0.f ? p.softmax_scale : (float)(1.0 / sqrt((double)p.head_dim));
    cudaError_t e = launch_decode(io, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "decode attention launch");
    return KVEC_OK;
}

kvec_status kvec_debug_scores(kvec_handle* h, kvec_debug_view* out) {
    if (!h || !out) return fail(KVEC_ERR_INVALID_ARG, "NULL argument");
    const Slot& sl = h->slots[h->last_slot];
    out->P_O = sl.PO;
    out->P_Oext = sl.POe;
    out->I = sl.I;
    out->sigma = sl.sigma;
    out->htop = sl.htop;
    out->pres_bits = sl.pres;
    out->Pprime = sl.Pprime;
    out->row_stats = reinterpret_cast<const float*>(h->rowstat_slot[h->last_slot]);
    out->max_seqlen = (int)row_stride(h->p.max_seqlen);
    out->words_per_row = h->words;
    return KVEC_OK;
}

kvec_status kvec_sync_status(kvec_handle* h) {
    if (!h) return fail(KVEC_ERR_INVALID_ARG, "handle is NULL");
    int prev = 0;
    kvec_status s = set_device(h, &prev);
    if (s != KVEC_OK) return s;
    DeviceGuard guard{prev, h->device};
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
    int err = 0;
    e = cudaMemcpy(&err, h->sc.err, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "reading the device error word");
    if (err) {
        cudaMemset(h->sc.err, 0, sizeof(int));
        return device_error_status(err);
    }
    return KVEC_OK;
}

void kvec_set_test_fault(int fault) { g_test_fault.store(fault == 1 ? 1 : 0, std::memory_order_relaxed); }

kvec_status kvec_set_profiling(kvec_handle* h, int enable) {
    if (!h) return fail(KVEC_ERR_INVALID_ARG, "handle is NULL");
    cudaDeviceSynchronize();
    recycle_timed(h);
    h->profiling = enable != 0;
    return KVEC_OK;
}

kvec_status kvec_kernel_time(kvec_handle* h, int kernel, double* total_ms, int* launches) {
    if (!h || !total_ms || !launches) return fail(KVEC_ERR_INVALID_ARG, "NULL argument");
    if (kernel < 0 || kernel >= kKernelKinds) return fail(KVEC_ERR_INVALID_ARG, "kernel id %d unknown", kernel);
    double sum = 0.0;
    int n = 0;
    for (auto& t : h->timed) {
        if (t.kind != kernel) continue;
        cudaError_t e = cudaEventSynchronize(t.stop);
        if (e != cudaSuccess) return cuda_fail(e, "cudaEventSynchronize");
        float ms = 0.f;
        e = cudaEventElapsedTime(&ms, t.start, t.stop);
        if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
        sum += ms;
        ++n;
    }
    *total_ms = sum;
    *launches = n;
    return KVEC_OK;
}

const char* kvec_status_string(kvec_status s) {
    switch (s) {
        case KVEC_OK: return "ok";
        case KVEC_ERR_INVALID_ARG: return "invalid argument";
        case KVEC_ERR_UNSUPPORTED: return "unsupported configuration";
        case KVEC_ERR_CUDA: return "CUDA error";
        case KVEC_ERR_DEVICE_TIMEOUT: return "device-side wait timed out";
        case KVEC_ERR_OOM: return "out of device memory";
    }
    return "unknown status";
}

const char* kvec_last_error(void) { return g_last_error.c_str(); }

}  // extern "C"
