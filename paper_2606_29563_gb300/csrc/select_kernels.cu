// Cross-head choice, preserved tokens, coverage-adjusted top-B and the
// coverage-state update (Section 4.1, Section 4.2, Algorithm 1), plus the K/V
// gather into the budget-sized cache.
//
// Top-k is an exact block-wide MSB radix select over order-preserving uint32
// keys (11/11/10-bit digits, shared-memory histograms, block scans built from
// warp shuffles and ballots).  Ties at the threshold go to the lower position.
#include <cooperative_groups.h>

#include "kvec_internal.cuh"

namespace cg = cooperative_groups;

namespace kvec {

namespace {

constexpr int kSmemKeys = 40960;   // positions whose keys fit in shared memory (160 KB)

__host__ __device__ inline bool keys_in_smem(int ML) { return ML <= kSmemKeys; }

struct TopkShared {
    int hist[2048];
    int wsum[32];
    int bcast[4];
};

// Exclusive prefix sum over the block (blockDim.x a multiple of 32, <= 1024).
__device__ int block_exclusive_sum(int v, int* wsum, int& total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int x = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, off);
        if (lane >= off) x += y;
    }
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int ws = lane < nw ? wsum[lane] : 0;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, ws, off);
            if (lane >= off) ws += y;
        }
        wsum[lane] = ws;
    }
    __syncthreads();
    const int before = warp ? wsum[warp - 1] : 0;
    total = wsum[nw - 1];
    __syncthreads();
    return before + x - v;
}

// ORs into bits[] (shared, one bit per position) the k largest keys of keys[0, n).
// Key 0 marks an ineligible position; the caller guarantees k <= #eligible.
__device__ void block_topk(const uint32_t* __restrict__ keys, int n, int k, uint32_t* bits, TopkShared& sm) {
    if (k <= 0 || n <= 0) return;
    const int tid = threadIdx.x, NT = blockDim.x;
    uint32_t prefix = 0, mask = 0;
    int kk = k;
    bool whole_bin = false;
    for (int pass = 0; pass < 3; ++pass) {
        const int sh = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
        const int nb = pass == 2 ? 1024 : 2048;
        for (int i = tid; i < nb; i += NT) sm.hist[i] = 0;
        __syncthreads();
        for (int t = tid; t < n; t += NT) {
            const uint32_t u = keys[t];
            if (u != 0u && (u & mask) == prefix) atomicAdd(&sm.hist[(u >> sh) & (nb - 1)], 1);
        }
        __syncthreads();
        // Thread i owns the i-th block of bins counted from the top.
        const int bpt = (nb + NT - 1) / NT;
        const int hi = nb - tid * bpt, lo = max(hi - bpt, 0);
        int mine = 0;
        for (int b = lo; b < hi; ++b) mine += sm.hist[b];
        int total;
        const int above_me = block_exclusive_sum(mine, sm.wsum, total);
        if (hi > 0 && above_me < kk && above_me + mine >= kk) {
            int acc = above_me;
            for (int b = hi - 1; b >= lo; --b) {
                if (acc + sm.hist[b] >= kk) {
                    sm.bcast[0] = b;
                    sm.bcast[1] = acc;
                    sm.bcast[2] = sm.hist[b];
                    break;
                }
                acc += sm.hist[b];
            }
        }
        __syncthreads();
        const int D = sm.bcast[0], above = sm.bcast[1], cnt = sm.bcast[2];
        __syncthreads();
        prefix |= (uint32_t)D << sh;
        mask |= (uint32_t)(nb - 1) << sh;
        kk -= above;
        if (cnt == kk) {
            whole_bin = true;
            break;
        }
    }
    // Positions strictly above the threshold prefix are in; positions equal to it
    // are in either all together or, when equal keys exceed the need, lowest first.
    const int nchunks = (n + NT - 1) / NT;
    int taken = 0;
    for (int ch = 0; ch < nchunks; ++ch) {
        const int t = ch * NT + tid;
        const uint32_t u = t < n ? keys[t] : 0u;
        const bool above = u != 0u && (u & mask) > prefix;
        const bool eq = u != 0u && (u & mask) == prefix;
        bool sel;
        if (whole_bin) {
            sel = above || eq;
        } else {
            int tot;
            const int r = block_exclusive_sum(eq ? 1 : 0, sm.wsum, tot);
            sel = above || (eq && taken + r < kk);
            taken += tot;
        }
        const unsigned bal = __ballot_sync(0xffffffffu, sel);
        if ((tid & 31) == 0 && bal) bits[(ch * NT + (tid & ~31)) >> 5] |= bal;
    }
    __syncthreads();
}

__device__ __forceinline__ uint32_t range_bits(int word, int lo, int hi) {
    // Bits of `word` covering positions in [lo, hi).
    const int b0 = word * 32;
    const int a = max(lo - b0, 0), e = min(hi - b0, 32);
    if (e <= a) return 0u;
    const uint32_t upto = e == 32 ? 0xffffffffu : ((1u << e) - 1u);
    return upto & ~((1u << a) - 1u);
}

// Max-pool (width 2*halo+1, stride 1, neighbours outside [0, Lc) ignored) of
// the four positions [t4, t4+4) of a row: the raw values [t4-8, t4+12) arrive
// as five float4 loads issued together.
struct Pooled4 {
    float v[4];
};

__device__ __forceinline__ Pooled4 pool4(const float* __restrict__ raw, int t4, int Lc, int halo) {
    float x[20];
#pragma unroll
    for (int b = 0; b < 5; ++b) {
        const int p = t4 - 8 + 4 * b;
        float4 f = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
        if (p >= 0 && p < Lc) f = __ldcg(reinterpret_cast<const float4*>(raw + p));
        x[4 * b] = p < Lc ? f.x : -INFINITY;
        x[4 * b + 1] = p + 1 < Lc ? f.y : -INFINITY;
        x[4 * b + 2] = p + 2 < Lc ? f.z : -INFINITY;
        x[4 * b + 3] = p + 3 < Lc ? f.w : -INFINITY;
    }
    Pooled4 out;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float m = x[8 + i];
#pragma unroll
        for (int d = 1; d <= kMaxPool / 2; ++d)
            if (d <= halo) m = fmaxf(m, fmaxf(x[8 + i - d], x[8 + i + d]));
        out.v[i] = m;
    }
    return out;
}

// Running (count, mean, sum of squared deviations); merge() is Chan et al.'s
// pairwise update, stable in fp32 (no cancellation of sum(x^2) - n*mean^2).
struct Moments {
    float n, mean, m2;
    __device__ void add(float x) {
        n += 1.f;
        const float d = x - mean;
        mean += d / n;
        m2 += d * (x - mean);
    }
    __device__ void merge(float nb, float meanb, float m2b) {
        if (nb == 0.f) return;
        if (n == 0.f) {
            n = nb;
            mean = meanb;
            m2 = m2b;
            return;
        }
        const float nt = n + nb, d = meanb - mean;
        mean += d * (nb / nt);
        m2 += m2b + d * d * (n * nb / nt);
        n = nt;
    }
};

__device__ Moments block_moments(Moments v, float3* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    for (int off = 16; off; off >>= 1)
        v.merge(__shfl_xor_sync(0xffffffffu, v.n, off), __shfl_xor_sync(0xffffffffu, v.mean, off),
                __shfl_xor_sync(0xffffffffu, v.m2, off));
    if (lane == 0) red[warp] = make_float3(v.n, v.mean, v.m2);
    __syncthreads();
    Moments t{0.f, 0.f, 0.f};
    if (lane < nw) t = Moments{red[lane].x, red[lane].y, red[lane].z};
    for (int off = 16; off; off >>= 1)
        t.merge(__shfl_xor_sync(0xffffffffu, t.n, off), __shfl_xor_sync(0xffffffffu, t.mean, off),
                __shfl_xor_sync(0xffffffffu, t.m2, off));
    __syncthreads();
    return t;
}

// Section 4.1 and the preserved tokens of Section 4.2.  One thread-block
// cluster per sequence, one CTA per KV head (cluster rank = head):
//   pool the head's P_O and P_O' rows and a slice of I (max-pool, inherited
//   from SnapKV), sigma_h = sample std of pooled P_O over the candidates
//   (Welford/Chan moments in fp32), exchange sigma through distributed shared memory, the
//   delta lowest-sigma heads take the O' scores, then the top-K preserved
//   tokens of the chosen row by radix select.
__global__ void __launch_bounds__(kSelectThreads) heads_kernel(Geometry G, LayerIO io, Scratch sc, Slot sl) {
    cg::cluster_group cluster = cg::this_cluster();
    __shared__ TopkShared sm;
    __shared__ float3 red[32];
    __shared__ float sig_self;
    extern __shared__ uint32_t bits[];
    const int h = (int)cluster.block_rank(), s = blockIdx.y;
    const int tid = threadIdx.x, NT = blockDim.x;
    const int L = io.cu[s + 1] - io.cu[s];
    const int Lc = L - G.w;
    const int halo = G.pool / 2;
    const size_t row = (size_t)s * G.Hkv + h;
    // Pool P_O and P_O' of this head (four positions per thread per step) and
    // accumulate the sums of pooled P_O and of its squares in fp64.
    Moments mom{0.f, 0.f, 0.f};
    const float* rO = sl.rawO + row * G.ML;
    const float* rOe = sl.rawOe + row * G.ML;
    for (int t4 = 4 * tid; t4 < Lc; t4 += 4 * NT) {
        const Pooled4 a = pool4(rO, t4, Lc, halo);
        const Pooled4 b = pool4(rOe, t4, Lc, halo);
        *reinterpret_cast<float4*>(sl.PO + row * G.ML + t4) = make_float4(a.v[0], a.v[1], a.v[2], a.v[3]);
        *reinterpret_cast<float4*>(sl.POe + row * G.ML + t4) = make_float4(b.v[0], b.v[1], b.v[2], b.v[3]);
#pragma unroll
        for (int i = 0; i < 4; ++i)
            if (t4 + i < Lc) mom.add(a.v[i]);
    }
    // This CTA's slice of pooled I.
    {
        const int per = ((Lc + G.Hkv - 1) / G.Hkv + 3) & ~3;
        const int a0 = min(h * per, Lc), b0 = min(a0 + per, Lc);
        const float* rI = sl.rawI + (size_t)s * G.ML;
        for (int t4 = a0 + 4 * tid; t4 < b0; t4 += 4 * NT) {
            const Pooled4 c = pool4(rI, t4, Lc, halo);
            *reinterpret_cast<float4*>(sl.I + (size_t)s * G.ML + t4) = make_float4(c.v[0], c.v[1], c.v[2], c.v[3]);
        }
    }
    mom = block_moments(mom, red);
    const float sigma = Lc >= 2 ? sqrtf(fmaxf(mom.m2, 0.f) / (float)(Lc - 1)) : 0.f;
    if (tid == 0) sig_self = sigma;
    for (int wd = tid; wd < G.words; wd += NT) bits[wd] = 0u;
    cluster.sync();
    __shared__ int top_flag;
    if (tid < 32) {
        const float so = tid < G.Hkv ? *cluster.map_shared_rank(&sig_self, tid) : INFINITY;
        const bool before = tid < G.Hkv && (so < sigma || (so == sigma && tid < h));
        const int rank = __popc(__ballot_sync(0xffffffffu, before));
        if (tid == 0) top_flag = rank < G.delta;
    }
    __syncthreads();
    const int top = top_flag;
    if (tid == 0) {
        sl.sigma[row] = sigma;
        sl.htop[row] = top;
    }
    if (L > G.budget && G.Kp > 0) {
        const float* __restrict__ P = (top ? sl.POe : sl.PO) + row * G.ML;
        uint32_t* keys = keys_in_smem(G.ML) ? bits + G.words : sc.keys + row * G.ML;
        for (int b0 = 4 * tid; b0 < Lc; b0 += 16 * NT) {
            float4 pv[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int t4 = b0 + 4 * u * NT;
                pv[u] = t4 < Lc ? __ldcg(reinterpret_cast<const float4*>(P + t4)) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int t4 = b0 + 4 * u * NT;
                const float x[4] = {pv[u].x, pv[u].y, pv[u].z, pv[u].w};
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    if (t4 + i < Lc) keys[t4 + i] = float_order_key(x[i]);
            }
        }
        __syncthreads();
        block_topk(keys, Lc, G.Kp, bits, sm);
    }
    uint32_t* pres = sl.pres + row * G.words;
    for (int wd = tid; wd < G.words; wd += NT) pres[wd] = bits[wd];
    cluster.sync();   // peers may still read sig_self
}

// Section 4.2: P' = P + lambda * I * (1 - n_t / (l + 1)); the preserved tokens
// stay, the rest of B - w goes to the largest P'; the last w tokens are kept.
// Writes out_idx (ascending) and folds the union of all heads into n_t once the
// last head of the sequence is done.  Grid (Hkv, batch).
__global__ void __launch_bounds__(kSelectThreads) select_kernel(Geometry G, LayerIO io, Scratch sc, Slot sl) {
    __shared__ TopkShared sm;
    __shared__ int last_head;
    extern __shared__ uint32_t bits[];
    const int h = blockIdx.x, s = blockIdx.y;
    const int tid = threadIdx.x, NT = blockDim.x;
    const int L = io.cu[s + 1] - io.cu[s];
    const int Lc = L - G.w;
    const int wordsL = (L + 31) >> 5;
    uint8_t* st = io.state + (size_t)s * G.state_stride;
    const uint32_t ell = reinterpret_cast<const uint32_t*>(st)[0];
    uint8_t* ncount = st + G.state_n_off;
    if (ell >= 255u) {  // n_t is 8-bit: a state that already saw 255 layers cannot count another
        if (tid == 0) atomicExch(sc.err, 2);
        return;
    }
    for (int wd = tid; wd < G.words; wd += NT) bits[wd] = 0u;
    __syncthreads();
    if (L > G.budget) {
        const size_t row = (size_t)s * G.Hkv + h;
        const int top = sl.htop[row];
        const float* P = (top ? sl.POe : sl.PO) + row * G.ML;
        const float* I = sl.I + (size_t)s * G.ML;
        const uint32_t* pres = sl.pres + row * G.words;
        float* Pp = sl.Pprime + row * G.ML;
        uint32_t* keys = keys_in_smem(G.ML) ? bits + G.words : sc.keys_sel + row * G.ML;
        const float denom = (float)(ell + 1u);
        for (int b0 = 4 * tid; b0 < Lc; b0 += 8 * NT) {
            float4 pv[2], iv[2];
            uchar4 nv[2];
            uint32_t pw[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int t4 = b0 + 4 * u * NT;
                if (t4 < Lc) {
                    pv[u] = *reinterpret_cast<const float4*>(P + t4);
                    iv[u] = *reinterpret_cast<const float4*>(I + t4);
                    nv[u] = *reinterpret_cast<const uchar4*>(ncount + t4);
                    pw[u] = pres[t4 >> 5];
                }
            }
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int t4 = b0 + 4 * u * NT;
                if (t4 >= Lc) continue;
                const float p4[4] = {pv[u].x, pv[u].y, pv[u].z, pv[u].w};
                const float i4[4] = {iv[u].x, iv[u].y, iv[u].z, iv[u].w};
                const uint8_t n4[4] = {nv[u].x, nv[u].y, nv[u].z, nv[u].w};
                float out[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int t = t4 + i;
                    const float coverage = (float)n4[i] / denom;
                    const float pp = p4[i] + G.lambda * (i4[i] * (1.f - coverage));
                    out[i] = pp;
                    const bool kept = (pw[u] >> (t & 31)) & 1u;
                    if (t < Lc) keys[t] = kept ? 0u : float_order_key(pp);
                }
                *reinterpret_cast<float4*>(Pp + t4) = make_float4(out[0], out[1], out[2], out[3]);
            }
        }
        __syncthreads();
        block_topk(keys, Lc, G.k2, bits, sm);
        for (int wd = tid; wd < wordsL; wd += NT) bits[wd] |= pres[wd] | range_bits(wd, Lc, L);
    } else {
        for (int wd = tid; wd < wordsL; wd += NT) bits[wd] = range_bits(wd, 0, L);
    }
    __syncthreads();

    // Ascending positions: each thread owns a contiguous run of words.
    int32_t* oi = io.out_idx + ((size_t)s * G.Hkv + h) * G.budget;
    const int wpt = (wordsL + NT - 1) / NT;
    const int w_lo = min(tid * wpt, wordsL), w_hi = min(w_lo + wpt, wordsL);
    int mine = 0;
    for (int wd = w_lo; wd < w_hi; ++wd) mine += __popc(bits[wd]);
    int total;
    int pos = block_exclusive_sum(mine, sm.wsum, total);
    for (int wd = w_lo; wd < w_hi; ++wd) {
        uint32_t b = bits[wd];
        while (b) {
            const int bit = __ffs(b) - 1;
            b &= b - 1u;
            if (pos < G.budget) oi[pos] = wd * 32 + bit;
            ++pos;
        }
    }
    for (int j = total + tid; j < G.budget; j += NT) oi[j] = -1;

    // Union over heads, then the last head of the sequence updates n_t (Section 4.2).
    uint32_t* ub = sc.ubits + (size_t)s * G.words;
    for (int wd = tid; wd < wordsL; wd += NT)
        if (bits[wd]) atomicOr(&ub[wd], bits[wd]);
    __threadfence();
    __syncthreads();
    if (tid == 0) last_head = atomicAdd(&sc.ucount[s], 1u) == (unsigned)(G.Hkv - 1);
    __syncthreads();
    if (!last_head) return;
    __threadfence();
    for (int t4 = 4 * tid; t4 < L; t4 += 4 * NT) {
        const uint32_t wv = __ldcg(&ub[t4 >> 5]) >> (t4 & 31);
        uchar4 n4 = *reinterpret_cast<uchar4*>(ncount + t4);
        n4.x = (uint8_t)(n4.x + (wv & 1u));
        if (t4 + 1 < L) n4.y = (uint8_t)(n4.y + ((wv >> 1) & 1u));
        if (t4 + 2 < L) n4.z = (uint8_t)(n4.z + ((wv >> 2) & 1u));
        if (t4 + 3 < L) n4.w = (uint8_t)(n4.w + ((wv >> 3) & 1u));
        *reinterpret_cast<uchar4*>(ncount + t4) = n4;
    }
    __syncthreads();
    uint32_t* last_union = reinterpret_cast<uint32_t*>(st + G.state_union_off);
    for (int wd = tid; wd < G.words; wd += NT) {
        last_union[wd] = __ldcg(&ub[wd]);
        ub[wd] = 0u;
    }
    if (tid == 0) {
        reinterpret_cast<uint32_t*>(st)[0] = ell + 1u;
        reinterpret_cast<uint32_t*>(st)[1] = (uint32_t)L;
        sc.ucount[s] = 0u;
    }
}

// out_k[s,h,j,:] = K[cu[s] + idx[s,h,j], h, :] (zeros for idx = -1); the same for V.
// Grid (ceil(B/16), Hkv, batch), 256 threads: a half-warp moves one 256-byte row.
__global__ void __launch_bounds__(256) gather_kernel(Geometry G, LayerIO io) {
    const int s = blockIdx.z, h = blockIdx.y;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int row = blockIdx.x * 16 + warp * 2 + (lane >> 4), sub = lane & 15;
    if (row >= G.budget) return;
    const size_t orow = ((size_t)s * G.Hkv + h) * G.budget + row;
    const int idx = io.out_idx[orow];
    const int L = io.cu[s + 1] - io.cu[s];
    uint4 kv = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
    if (idx >= 0 && idx < L) {
        const size_t src = (((size_t)io.cu[s] + idx) * G.Hkv + h) * kHeadDim + sub * 8;
        kv = __ldg(reinterpret_cast<const uint4*>(io.k + src));
        vv = __ldg(reinterpret_cast<const uint4*>(io.v + src));
    }
    reinterpret_cast<uint4*>(io.out_k + orow * kHeadDim)[sub] = kv;
    reinterpret_cast<uint4*>(io.out_v + orow * kHeadDim)[sub] = vv;
}

}  // namespace

size_t select_smem_bytes(const Geometry& g) {
    return sizeof(uint32_t) * ((size_t)g.words + (keys_in_smem(g.ML) ? (size_t)g.ML : 0));
}

size_t heads_smem_bytes(const Geometry& g) { return select_smem_bytes(g); }

cudaError_t configure_select() {
    const int need = (int)(sizeof(uint32_t) * (kSmemKeys + kSmemKeys / 32));
    cudaError_t e = cudaFuncSetAttribute(heads_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, need);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(heads_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, need);
    return e;
}

cudaError_t launch_heads(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(g.Hkv, g.batch);
    cfg.blockDim = dim3(kSelectThreads);
    cfg.dynamicSmemBytes = heads_smem_bytes(g);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = g.Hkv;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, heads_kernel, g, io, sc, sl);
}

void launch_select(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st) {
    select_kernel<<<dim3(g.Hkv, g.batch), kSelectThreads, select_smem_bytes(g), st>>>(g, io, sc, sl);
}

void launch_gather(const Geometry& g, const LayerIO& io, cudaStream_t st) {
    gather_kernel<<<dim3((g.budget + 15) / 16, g.Hkv, g.batch), 256, 0, st>>>(g, io);
}

}  // namespace kvec
