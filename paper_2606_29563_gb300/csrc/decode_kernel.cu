// One decoding step of attention over the compacted KV cache that the
// selection leaves behind.  Section 4.1: after the per-head top-B selection the
// keys and values of the kept tokens are the cache the subsequent decoding
// steps read; Section 5.3 measures decoding over it.  For sequence s and query
// head hq (KV head h = hq / g):
//   out[s][hq] = sum_{j < n_s} softmax_j(scale * <q[s][hq], k[s][h][j]>) v[s][h][j].
//
// The work is a few MB of K/V rows per call, read once: HBM- and latency-bound,
// no dense contraction worth the tensor cores (g <= 8 query rows per KV head).
// Split-K over the cache inside one thread-block cluster per (s, h): each of
// the kDecSplits CTAs streams its range of cached rows through shared memory in
// 64-row tiles and keeps an online (max, sum, output) per query head; after a
// cluster barrier, CTA r merges query head r from every CTA's shared memory
// (distributed shared memory), so one launch does the whole step.
#include "kvec_internal.cuh"
#include "sm100_ptx.cuh"

#include <cooperative_groups.h>

namespace kvec {

namespace {

namespace cg = cooperative_groups;

constexpr int kDecTile = 64;                     // cached rows per shared-memory tile
constexpr int kDecThreads = 256;
constexpr int kDecMaxG = 8;                      // query heads per KV head
constexpr int kDecSplits = 8;                    // CTAs per (sequence, KV head): one cluster
constexpr int kKRowHalves = kHeadDim + 8;        // K row stride in bf16 (16-byte pad: no bank conflicts)

struct DecArgs {
    const __nv_bfloat16* q;      // [batch][Hq][d]
    const __nv_bfloat16* k;      // [batch][Hkv][cap][d]
    const __nv_bfloat16* v;
    const int* lens;             // [batch]
    float* out;                  // [batch][Hq][d]
    int Hq, Hkv, g, cap, chunk;
    float sl2;                   // softmax scale * log2(e)
};

__global__ void __launch_bounds__(kDecThreads) decode_kernel(const __grid_constant__ DecArgs A) {
    __shared__ __align__(16) float qs[kDecMaxG][kHeadDim];   // the group's queries; later this CTA's outputs
    __shared__ __align__(16) __nv_bfloat16 ks[kDecTile][kKRowHalves];
    __shared__ __align__(16) __nv_bfloat16 vs[kDecTile][kHeadDim];
    __shared__ float ps[kDecMaxG][kDecTile];
    __shared__ float m_run[kDecMaxG], l_run[kDecMaxG], corr[kDecMaxG];
    cg::cluster_group cluster = cg::this_cluster();
    const int sp = (int)cluster.block_rank(), h = blockIdx.y, s = blockIdx.z;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int g = A.g, cap = A.cap;
    const int n = min(max(__ldg(&A.lens[s]), 0), cap);
    const int t_begin = sp * A.chunk, t_end = min(n, t_begin + A.chunk);
    const size_t kv_base = ((size_t)s * A.Hkv + h) * (size_t)cap * kHeadDim;
    const __nv_bfloat16* kg = A.k + kv_base;
    const __nv_bfloat16* vg = A.v + kv_base;

    // The group's query rows, widened to fp32.
    for (int i = tid; i < g * kHeadDim; i += kDecThreads) {
        const int j = i / kHeadDim, c = i - j * kHeadDim;
        qs[j][c] = __bfloat162float(A.q[((size_t)s * A.Hq + h * g + j) * kHeadDim + c]);
    }
    if (tid < kDecMaxG) {
        m_run[tid] = -INFINITY;
        l_run[tid] = 0.f;
    }
    // Output pairs of this thread: (query head j, columns 2*dp, 2*dp + 1) for
    // idx = tid and tid + 256 (g * 64 <= 512 pairs).
    float acc[2][2] = {{0.f, 0.f}, {0.f, 0.f}};

    for (int t0 = t_begin; t0 < t_end; t0 += kDecTile) {
        const int nt = min(kDecTile, t_end - t0);
        __syncthreads();   // the previous tile is consumed; qs and the running values are set
        // K and V rows of the tile: 16-byte pieces, 16 per row.
        for (int i = tid; i < nt * 16; i += kDecThreads) {
            const int r = i >> 4, c = (i & 15) * 8;
            const size_t gofs = (size_t)(t0 + r) * kHeadDim + c;
            *reinterpret_cast<uint4*>(&ks[r][c]) = __ldg(reinterpret_cast<const uint4*>(kg + gofs));
            *reinterpret_cast<uint4*>(&vs[r][c]) = __ldg(reinterpret_cast<const uint4*>(vg + gofs));
        }
        __syncthreads();
        // Logits in log2 units, one (query head, row) per thread and pass.
        for (int i = tid; i < g * kDecTile; i += kDecThreads) {
            const int j = i / kDecTile, r = i - j * kDecTile;
            float x = -INFINITY;
            if (r < nt) {
                float d0 = 0.f, d1 = 0.f;
#pragma unroll
                for (int c = 0; c < kHeadDim; c += 8) {
                    const uint4 kw = *reinterpret_cast<const uint4*>(&ks[r][c]);
                    const __nv_bfloat162* k2 = reinterpret_cast<const __nv_bfloat162*>(&kw);
                    const float4 qa = *reinterpret_cast<const float4*>(&qs[j][c]);
                    const float4 qb = *reinterpret_cast<const float4*>(&qs[j][c + 4]);
                    const float2 k01 = __bfloat1622float2(k2[0]), k23 = __bfloat1622float2(k2[1]);
                    const float2 k45 = __bfloat1622float2(k2[2]), k67 = __bfloat1622float2(k2[3]);
                    d0 = fmaf(qa.x, k01.x, d0);
                    d1 = fmaf(qa.y, k01.y, d1);
                    d0 = fmaf(qa.z, k23.x, d0);
                    d1 = fmaf(qa.w, k23.y, d1);
                    d0 = fmaf(qb.x, k45.x, d0);
                    d1 = fmaf(qb.y, k45.y, d1);
                    d0 = fmaf(qb.z, k67.x, d0);
                    d1 = fmaf(qb.w, k67.y, d1);
                }
                x = (d0 + d1) * A.sl2;
            }
            ps[j][r] = x;
        }
        __syncthreads();
        // Online softmax of each query head (warp j): new maximum, the old sums'
        // correction, the tile's weights 2^(x - m).
        if (warp < g) {
            const int j = warp;
            const float x0 = ps[j][lane], x1 = ps[j][lane + 32];
            float mt = fmaxf(x0, x1);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, o));
            const float m_old = m_run[j];
            const float m_new = fmaxf(m_old, mt);   // finite: the tile has a valid row
            const float p0 = ptx::ex2(x0 - m_new), p1 = ptx::ex2(x1 - m_new);
            ps[j][lane] = p0;
            ps[j][lane + 32] = p1;
            float sum = p0 + p1;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
            __syncwarp();
            if (lane == 0) {
                const float c = ptx::ex2(m_old - m_new);   // 0 while m_old is -inf
                corr[j] = c;
                l_run[j] = l_run[j] * c + sum;
                m_run[j] = m_new;
            }
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const int idx = tid + k * kDecThreads;
            const int j = idx >> 6, dp = idx & 63;
            if (j < g) {
                const float c = corr[j];
                float a0 = acc[k][0] * c, a1 = acc[k][1] * c;
                for (int r = 0; r < nt; ++r) {
                    const float p = ps[j][r];
                    const float2 vv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&vs[r][2 * dp]));
                    a0 = fmaf(p, vv.x, a0);
                    a1 = fmaf(p, vv.y, a1);
                }
                acc[k][0] = a0;
                acc[k][1] = a1;
            }
        }
    }
    // This CTA's unnormalised outputs replace the queries in shared memory; its
    // (max, sum) per query head stay in m_run / l_run.
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int idx = tid + k * kDecThreads;
        const int j = idx >> 6, dp = idx & 63;
        if (j < g) *reinterpret_cast<float2*>(&qs[j][2 * dp]) = make_float2(acc[k][0], acc[k][1]);
    }
    cluster.sync();
    // CTA r merges query head r over the cluster:
    // out = sum_c 2^(m_c - M) o_c / sum_c 2^(m_c - M) l_c, zeros for an empty cache.
    if (sp < g && tid < kHeadDim) {
        const int j = sp;
        float M = -INFINITY;
#pragma unroll
        for (int c = 0; c < kDecSplits; ++c) M = fmaxf(M, *cluster.map_shared_rank(&m_run[j], c));
        float L = 0.f, O = 0.f;
        if (M != -INFINITY) {
#pragma unroll
            for (int c = 0; c < kDecSplits; ++c) {
                const float m = *cluster.map_shared_rank(&m_run[j], c);
                if (m == -INFINITY) continue;
                const float w = ptx::ex2(m - M);
                L = fmaf(w, *cluster.map_shared_rank(&l_run[j], c), L);
                O = fmaf(w, *cluster.map_shared_rank(&qs[j][tid], c), O);
            }
        }
        A.out[((size_t)s * A.Hq + h * g + j) * kHeadDim + tid] = L > 0.f ? O / L : 0.f;
    }
    cluster.sync();   // no CTA leaves while another still reads its shared memory
}

}  // namespace

cudaError_t launch_decode(const DecodeIO& io, cudaStream_t st) {
    DecArgs a{};
    a.q = io.q;
    a.k = io.k;
    a.v = io.v;
    a.lens = io.lens;
    a.out = io.out;
    a.Hq = io.Hq;
    a.Hkv = io.Hkv;
    a.g = io.Hq / io.Hkv;
    a.cap = io.cap;
    const int per = (io.cap + kDecSplits - 1) / kDecSplits;
    a.chunk = (per + kDecTile - 1) / kDecTile * kDecTile;
    a.sl2 = io.scale * 1.4426950408889634f;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kDecSplits, io.Hkv, io.batch);
    cfg.blockDim = dim3(kDecThreads);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kDecSplits;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, decode_kernel, a);
}

}  // namespace kvec
