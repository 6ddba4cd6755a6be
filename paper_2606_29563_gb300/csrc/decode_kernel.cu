// One decoding step of attention over the compacted KV cache that the
// selection leaves behind.  Section 4.1: after the per-head top-B selection the
// keys and values of the kept tokens are the cache the subsequent decoding
// steps read; Section 5.3 measures decoding over it.  For sequence s and query
// head hq (KV head h = hq / g):
//   out[s][hq] = sum_{j < n_s} softmax_j(scale * <q[s][hq], k[s][h][j]>) v[s][h][j].
//
// The work is a few MB of K/V rows per call, read once: HBM- and latency-bound,
// no dense contraction worth the tensor cores (g <= 8 query rows per KV head).
// Split-K over the cache: CTA (split, h, s) streams its range of cached rows
// through shared memory in 64-row tiles and keeps an online (max, sum, output)
// for the g query heads of KV head h; a second kernel merges the splits.
#include "kvec_internal.cuh"
#include "sm100_ptx.cuh"

namespace kvec {

namespace {

constexpr int kDecTile = 64;                     // cached rows per shared-memory tile
constexpr int kDecThreads = 256;
constexpr int kDecMaxG = 8;                      // query heads per KV head
constexpr int kKRowHalves = kHeadDim + 8;        // K row stride in bf16 (16-byte pad: no bank conflicts)

struct DecArgs {
    const __nv_bfloat16* q;      // [batch][Hq][d]
    const __nv_bfloat16* k;      // [batch][Hkv][cap][d]
    const __nv_bfloat16* v;
    const int* lens;             // [batch]
    float* part;                 // [batch][Hq][nsplit][d]  unnormalised split outputs
    float2* ml;                  // [batch][Hq][nsplit]     split (max in log2 units, sum)
    float* out;                  // [batch][Hq][d]
    int Hq, Hkv, g, cap, nsplit, chunk;
    float sl2;                   // softmax scale * log2(e)
};

__global__ void __launch_bounds__(kDecThreads) decode_partial_kernel(const __grid_constant__ DecArgs A) {
    __shared__ __align__(16) float qs[kDecMaxG][kHeadDim];
    __shared__ __align__(16) __nv_bfloat16 ks[kDecTile][kKRowHalves];
    __shared__ __align__(16) __nv_bfloat16 vs[kDecTile][kHeadDim];
    __shared__ float ps[kDecMaxG][kDecTile];
    __shared__ float m_run[kDecMaxG], l_run[kDecMaxG], corr[kDecMaxG];
    if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    const int sp = blockIdx.x, h = blockIdx.y, s = blockIdx.z;
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
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int idx = tid + k * kDecThreads;
        const int j = idx >> 6, dp = idx & 63;
        if (j < g) {
            const size_t row = ((size_t)s * A.Hq + h * g + j) * A.nsplit + sp;
            *reinterpret_cast<float2*>(A.part + row * kHeadDim + 2 * dp) = make_float2(acc[k][0], acc[k][1]);
        }
    }
    if (tid < g) A.ml[((size_t)s * A.Hq + h * g + tid) * A.nsplit + sp] = make_float2(m_run[tid], l_run[tid]);
}

// out = sum_s 2^(m_s - M) o_s / sum_s 2^(m_s - M) l_s over the splits; zeros
// for an empty cache.  Grid (Hq, batch), one thread per output column.
__global__ void __launch_bounds__(kHeadDim) decode_combine_kernel(const __grid_constant__ DecArgs A) {
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    const int hq = blockIdx.x, s = blockIdx.y, c = threadIdx.x;
    const size_t row = ((size_t)s * A.Hq + hq) * A.nsplit;
    float M = -INFINITY;
    for (int sp = 0; sp < A.nsplit; ++sp) M = fmaxf(M, __ldcg(&A.ml[row + sp]).x);
    float L = 0.f, O = 0.f;
    if (M != -INFINITY) {
        for (int sp = 0; sp < A.nsplit; ++sp) {
            const float2 ml = __ldcg(&A.ml[row + sp]);
            if (ml.x == -INFINITY) continue;
            const float w = ptx::ex2(ml.x - M);
            L = fmaf(w, ml.y, L);
            O = fmaf(w, __ldcg(&A.part[(row + sp) * kHeadDim + c]), O);
        }
    }
    A.out[((size_t)s * A.Hq + hq) * kHeadDim + c] = L > 0.f ? O / L : 0.f;
}

}  // namespace

int decode_splits(int cap) {
    int ns = (cap + kDecTile - 1) / kDecTile;
    return ns < 1 ? 1 : (ns > kDecMaxSplits ? kDecMaxSplits : ns);
}

cudaError_t launch_decode(const DecodeIO& io, cudaStream_t st) {
    DecArgs a{};
    a.q = io.q;
    a.k = io.k;
    a.v = io.v;
    a.lens = io.lens;
    a.part = io.part;
    a.ml = io.ml;
    a.out = io.out;
    a.Hq = io.Hq;
    a.Hkv = io.Hkv;
    a.g = io.Hq / io.Hkv;
    a.cap = io.cap;
    a.nsplit = decode_splits(io.cap);
    const int per = (io.cap + a.nsplit - 1) / a.nsplit;
    a.chunk = (per + kDecTile - 1) / kDecTile * kDecTile;
    a.sl2 = io.scale * 1.4426950408889634f;
    decode_partial_kernel<<<dim3(a.nsplit, io.Hkv, io.batch), kDecThreads, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(io.Hq, io.batch);
    cfg.blockDim = dim3(kHeadDim);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, decode_combine_kernel, a);
}

}  // namespace kvec
