// Internal declarations of the K-VEC CUDA path (sm_103a).  Not part of the ABI.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace kvec {

constexpr int kHeadDim = 128;      // d supported by the score kernel
constexpr int kTileT = 128;        // tokens per score / window tile (one MMA N or M block)
constexpr int kMaxPool = 15;       // largest pool kernel (halo 7)
constexpr int kSelectThreads = 512;
constexpr int kMaxObsWindow = 64;  // largest O: the window kernel keeps O x 128 head maxima in shared memory
constexpr int kWinHeadsPerCta = 8; // KV heads one window CTA processes

// Sizes and hyper-parameters shared by every kernel of one call.
struct Geometry {
    int Hq, Hkv, g, w, O, Oe, pool, delta;
    int wk;            // kept tail: w, or 0 when every position is a candidate; candidates [0, L - wk)
    int pool_avg;      // 1: average pool instead of max-pool
    int head_entropy;  // 1: rank heads by minus the entropy of pooled P_O instead of its std
    int R;             // rows per KV head = g * w, ordered r = q * g + j
    float lambda;
    float sl2;         // softmax scale * log2(e)
    int ML;            // max_seqlen: row stride of per-position workspace arrays
    int words;         // ceil(ML / 32)
    int batch, budget, Kp, k2;
    int ada;           // 1: head-wise adaptive fill (a head ranks f0 of its k2 fill slots itself)
    int f0;            // fill slots a head takes by its own ranking (k2 for the uniform fill)
    int extras;        // fill slots ranked over all heads of a sequence together: Hkv * (k2 - f0)
    int cap;           // rows per KV head of the outputs: budget + (Hkv - 1) * (k2 - f0)
    int jpool;         // adaptive fill: candidates a head offers the joint ranking, min(extras, 32 * words)
    int jstride;       // adaptive fill: per-sequence stride of the joint candidate arrays
    int total_tiles;   // sum over sequences of ceil(L_s / kTileT)
    int win_tiles;     // sum over sequences of ceil((L_s - wk) / kTileT): candidate tiles
    int HG, NG;        // KV heads per window CTA, window CTAs per candidate tile
    int total_tokens;  // cu_seqlens[batch]
    const int* cu_host;  // host copy of cu_seqlens (host-side planning only; not for device code)
    size_t state_stride;
    size_t state_n_off, state_union_off;
    int nlen;          // bytes of one sequence's n_t array (round_up(max_seqlen, 16))
};

// Device workspace owned by the handle (one slot of per-layer score arrays).
struct Slot {
    float* rawO;          // [max_batch][Hkv][ML]  Eq. 1 scores, window O, before pooling
    float* rawOe;         // [max_batch][Hkv][ML]  window O', before pooling
    float* rawI;          // [max_batch][ML]       importance, before pooling
    float* PO;            // [max_batch][Hkv][ML]  pooled Eq. 1 scores, window O
    float* POe;           // [max_batch][Hkv][ML]  pooled, window O'
    float* I;             // [max_batch][ML]       pooled importance
    float* sigma;         // [max_batch][Hkv]
    int* htop;            // [max_batch][Hkv]
    uint32_t* pres;       // [max_batch][Hkv][words]
    float* Pprime;        // [max_batch][Hkv][ML]
    float* wpart;         // [win_tiles][NG][O][kTileT] per-group head maxima of G_h[q][t] (NG > 1)
    uint32_t* sel;        // [max_batch][Hkv][words]  kept positions of the layer, one bit each
};

struct Scratch {
    float2* segpart;      // [total_tiles * Hkv][R] per-CTA segment (max, sum), keyed by the segment's first item
    float2* rowstat;      // [max_batch][Hkv][R]    (row max in log2 units, softmax denominator), for inspection
    uint32_t* keys;       // [max_batch][Hkv][ML]   radix-select keys of the heads kernel
    uint32_t* keys_sel;   // [max_batch][Hkv][ML]   radix-select keys of the select kernel
    uint32_t* jkeys;      // [max_batch][jstride]   adaptive fill: the heads' joint candidates' keys (a key row)
    int32_t* jpos;        // [max_batch][jstride]   their positions (candidate i belongs to head i / jpool)
    uint32_t* jbits;      // [max_batch][jstride / 32] winners of the joint ranking, one bit per candidate
    uint8_t* nbuf;        // [max_batch][nlen]      second copy of n_t (the coverage counts alternate)
    int* err;             // device error word
};

struct LayerIO {
    const __nv_bfloat16* q;   // [batch][w][Hq][d]
    const __nv_bfloat16* k;   // [total][Hkv][d]
    const __nv_bfloat16* v;
    const int* cu;            // device cu_seqlens
    uint8_t* state;
    int32_t* out_idx;
    __nv_bfloat16* out_k;
    __nv_bfloat16* out_v;
    const float* lse;         // [batch][w][Hq] natural-log softmax denominators of the window rows, or null
};

// One decoding step over a compacted cache (decode_kernel.cu).
struct DecodeIO {
    const __nv_bfloat16* q;   // [batch][Hq][d]
    const __nv_bfloat16* k;   // [batch][Hkv][cap][d]
    const __nv_bfloat16* v;
    const int* lens;          // [batch] valid cached rows, clamped to [0, cap]
    float* out;               // [batch][Hq][d]
    int batch, Hq, Hkv, cap;
    float scale;              // softmax scale
};

// ---------------------------------------------------------------- helpers

__device__ __forceinline__ uint32_t float_order_key(float f) {
    // Monotone map of IEEE floats onto unsigned integers (larger float -> larger key).
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Finds (sequence, local index) of global item `gi` where sequence s owns
// count(s) consecutive items; also returns the first global item of s.
template <class CountFn>
__device__ __forceinline__ bool locate_item(int batch, int gi, CountFn count, int& s, int& local, int& base) {
    int acc = 0;
    for (int b = 0; b < batch; ++b) {
        int c = count(b);
        if (gi < acc + c) { s = b; local = gi - acc; base = acc; return true; }
        acc += c;
    }
    return false;
}

__host__ __device__ __forceinline__ int tiles_of(int L) { return (L + kTileT - 1) / kTileT; }

// ---------------------------------------------------------------- launchers

// Host-side launch description of the score kernel (tensor maps encoded ahead of the launch).
struct ScorePlan {
    CUtensorMap kmap, qmap;
    alignas(16) unsigned char args[512];
    int grid, threads, mb;   // mb: 128-row M-blocks per KV head
    int chunk;               // work items per claim of the score kernel (segment boundaries of its partials)
    size_t smem;
    int num_sms;             // SMs of the device (persistent grids are sized from it)
};
cudaError_t plan_score(const Geometry& g, const LayerIO& io, const Scratch& sc, int num_sms, ScorePlan* plan);
// after_own_launch: the stream's previous kernel is the previous layer's launch
// of the same kernel (the multi-stream layer pipeline); the launch may then
// overlap it (programmatic stream serialization), as it reads none of its results.
// claim: an int in device memory, zero before the launch (the CTAs count the
// work chunks they claim on it; the layer's launch_rowstat sets it back to
// zero once the score grid has completed); a distinct one for every launch in flight.
cudaError_t launch_score(const ScorePlan& plan, int* claim, cudaStream_t st, bool after_own_launch);
// (m_r, Z_r) from the score launch's partials.  programmatic: a programmatic
// dependent of the stream's previous kernel.  after_score: that kernel is this
// layer's score launch, waited for (griddepcontrol.wait) before the partials
// are read; without it the partials must come through a full dependency and the
// previous kernel (the layer pipeline's previous window grid) is not waited for.
cudaError_t launch_rowstat(const ScorePlan& plan, const Geometry& g, const LayerIO& io, const Scratch& sc,
                           int* claim, cudaStream_t st, bool programmatic, bool after_score);
// (m_r, Z_r) = (lse * log2(e), 1) from the caller's log-sum-exp (io.lse), in place
// of the score and row-statistics launches.  programmatic: as for launch_rowstat
// without after_score (it reads only the caller's input).
cudaError_t launch_rowstat_lse(const Geometry& g, const LayerIO& io, const Scratch& sc, cudaStream_t st,
                               bool programmatic);
cudaError_t launch_window(const ScorePlan& sp, const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl,
                          cudaStream_t st, bool after_own_launch);
// CTAs of the grid launch_window starts for this layer (0 without candidates);
// lse: the layer comes with the caller's log-sum-exp (io.lse).
int window_grid_size(const ScorePlan& sp, const Geometry& g, bool lse);
// Launches kernel<<<grid, block, smem, st>>> with a scheduling priority (lower
// numbers first; the range comes from cudaDeviceGetStreamPriorityRange) and,
// with `programmatic`, as a programmatic dependent of the stream's previous
// kernel: it may start once that grid triggers launch_dependents and must
// execute griddepcontrol.wait before it reads what that grid writes.
template <class... KArgs, class... Args>
cudaError_t launch_prio(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, int priority,
                        bool programmatic, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributePriority;
    attr[0].val.priority = priority;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = programmatic ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

cudaError_t launch_heads(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st,
                         int priority);
// lcall: the layer's index within a call of ncall layers (0 for the first);
// prev: the previous layer's slot (null for lcall = 0), whose kept-position
// bits give that layer's union.  The coverage counts alternate between the
// state and sc.nbuf; launch_finalize folds the last layer's union (from its
// slot) into the state.  programmatic: the stream's previous kernel is the
// previous layer's selection (the layer pipeline's chain stream, whose only
// other dependency is a full one on this layer's heads kernels); the grid then
// stages this layer's scores while that one drains and waits
// (griddepcontrol.wait) before reading the coverage counts.  Never set it when
// the stream's previous kernel wrote this layer's scores.
cudaError_t launch_select(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, const Slot* prev,
                          cudaStream_t st, int priority, int lcall, int ncall, bool programmatic);
cudaError_t launch_finalize(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& last, cudaStream_t st,
                            int priority, int ncall);
// Adaptive fill: the layer's extra fill slots over every head of a sequence,
// ranked together, ORed into the heads' kept bits.  A programmatic dependent of
// the layer's selection (it waits for it).
cudaError_t launch_ada(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st,
                       int priority, int ncall);
// out_idx from the slot's kept-position bits, then the K/V rows.
cudaError_t launch_decode(const DecodeIO& io, cudaStream_t st);
void launch_gather(const Geometry& g, const LayerIO& io, const Slot& sl, cudaStream_t st);

// Fault injected by kvec_set_test_fault (0: none), read when a kernel is launched.
int test_fault();

size_t score_smem_bytes(const Geometry& g);
size_t window_smem_bytes(const Geometry& g);
cudaError_t configure_score(const Geometry& g);
cudaError_t configure_window(const Geometry& g);
cudaError_t configure_select();

}  // namespace kvec
